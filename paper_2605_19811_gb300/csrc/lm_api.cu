// Host side of the C ABI declared in include/lionmuon.h: argument validation,
// parameter classification (vectors vs hidden matrices), shape groups for the
// grouped Newton-Schulz GEMMs, device tables, workspace, and the per-step
// launch sequence of Algorithm 1 (Lion step, or Muon step on t mod P == 0).
#include <algorithm>
#include <array>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <limits>
#include <map>
#include <string>
#include <tuple>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "lm_internal.h"

namespace lm {

static std::atomic<uint64_t> g_launches{0};
void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }
int device_slot() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return -1;
  return (dev >= 0 && dev < kMaxDevices) ? dev : -1;
}
uint64_t env_wait_limit_ns() {
  const char* v = std::getenv("LM_WAIT_LIMIT_NS");
  if (v == nullptr || *v == '\0') return kDefaultWaitNs;
  char* end = nullptr;
  const unsigned long long x = std::strtoull(v, &end, 10);
  return (end != nullptr && *end == '\0' && x > 0) ? (uint64_t)x : kDefaultWaitNs;
}

namespace {

thread_local std::string g_last_error;

lm_status fail(lm_status st, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
lm_status fail(lm_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}
lm_status cuda_fail(cudaError_t e, const char* what) {
  if (e == cudaErrorMemoryAllocation) return fail(LM_ERR_OOM, "%s: %s", what, cudaGetErrorString(e));
  return fail(LM_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}
#define LM_CUDA(call, what)                     \
  do {                                          \
    cudaError_t e_ = (call);                    \
    if (e_ != cudaSuccess) return cuda_fail(e_, what); \
  } while (0)

size_t dtype_size(lm_dtype d) { return d == LM_BF16 ? 2 : 4; }
bool valid_dtype(int d) { return d == LM_BF16 || d == LM_F32; }
int64_t numel(const lm_tensor& t) { return t.rows * t.cols; }
bool is_matrix(const lm_tensor& t) { return t.rows > 1 && t.cols > 1; }
size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

lm_status check_tensor(const lm_tensor* t, const char* what, int i) {
  if (t->rows < 0 || t->cols < 0)
    return fail(LM_ERR_INVALID_ARG, "%s[%d]: negative shape (%lld x %lld)", what, i,
                (long long)t->rows, (long long)t->cols);
  if (!valid_dtype(t->dtype)) return fail(LM_ERR_DTYPE, "%s[%d]: unsupported dtype %d", what, i, (int)t->dtype);
  if (numel(*t) > 0) {
    if (t->data == nullptr) return fail(LM_ERR_INVALID_ARG, "%s[%d]: NULL data", what, i);
    if (reinterpret_cast<uintptr_t>(t->data) % 16 != 0)
      return fail(LM_ERR_ALIGN, "%s[%d]: data pointer not 16-byte aligned", what, i);
  }
  return LM_OK;
}

// The tensor's data must be device (or managed) memory of device `dev`: a
// host pointer handed to a kernel would fault or read the wrong memory.
lm_status check_device_memory(const lm_tensor* t, const char* what, int i, int dev) {
  if (numel(*t) == 0) return LM_OK;
  cudaPointerAttributes a{};
  cudaError_t e = cudaPointerGetAttributes(&a, t->data);
  if (e != cudaSuccess) {
    cudaGetLastError();   // an unknown pointer is an argument error, not a sticky CUDA error
    return fail(LM_ERR_INVALID_ARG, "%s[%d]: not a CUDA pointer (%s)", what, i, cudaGetErrorString(e));
  }
  if (a.type != cudaMemoryTypeDevice && a.type != cudaMemoryTypeManaged)
    return fail(LM_ERR_INVALID_ARG, "%s[%d]: data is %s memory, not device memory", what, i,
                a.type == cudaMemoryTypeHost ? "page-locked host" : "unregistered host");
  if (a.type == cudaMemoryTypeDevice && a.device != dev)
    return fail(LM_ERR_INVALID_ARG, "%s[%d]: data lives on device %d, the call runs on device %d", what, i,
                a.device, dev);
  return LM_OK;
}

lm_status check_config(const lm_config* c) {
  auto finite = [](double x) { return std::isfinite(x); };
  if (!(c->beta1 >= 0.0 && c->beta1 < 1.0) || !(c->beta2 >= 0.0 && c->beta2 < 1.0))
    return fail(LM_ERR_INVALID_ARG, "beta1/beta2 must lie in [0, 1)");
  if (!finite(c->eta_muon) || !finite(c->eta_lion) || c->eta_muon < 0 || c->eta_lion < 0)
    return fail(LM_ERR_INVALID_ARG, "learning rates must be finite and >= 0");
  if (!finite(c->weight_decay) || c->weight_decay < 0) return fail(LM_ERR_INVALID_ARG, "weight_decay must be >= 0");
  if (c->period < 0) return fail(LM_ERR_INVALID_ARG, "period must be >= 0 (0 = infinity)");
  if (c->ns_steps < 0 || c->ns_steps > 64) return fail(LM_ERR_INVALID_ARG, "ns_steps must be in [0, 64]");
  if (!finite(c->ns_a) || !finite(c->ns_b) || !finite(c->ns_c)) return fail(LM_ERR_INVALID_ARG, "NS coefficients must be finite");
  if (c->ns_coeffs != nullptr)
    for (int k = 0; k < 3 * c->ns_steps; ++k)
      if (!finite(c->ns_coeffs[k])) return fail(LM_ERR_INVALID_ARG, "ns_coeffs[%d] is not finite", k);
  if (!finite(c->ns_eps) || c->ns_eps < 0) return fail(LM_ERR_INVALID_ARG, "ns_eps must be >= 0");
  if (!finite(c->shape_scale) || c->shape_scale < 0) return fail(LM_ERR_INVALID_ARG, "shape_scale must be >= 0");
  if (c->ns_precision != LM_BF16 && c->ns_precision != LM_F32 && c->ns_precision != LM_NS_F32_TC)
    return fail(LM_ERR_INVALID_ARG, "ns_precision must be LM_BF16, LM_F32 or LM_NS_F32_TC");
  if (c->schedule != LM_SCHEDULE_PERIOD && c->schedule != LM_SCHEDULE_STABLE_RANK)
    return fail(LM_ERR_INVALID_ARG, "schedule must be LM_SCHEDULE_PERIOD or LM_SCHEDULE_STABLE_RANK");
  if (c->schedule == LM_SCHEDULE_STABLE_RANK) {
    if (!finite(c->srank_alpha) || !(c->srank_alpha > 0)) return fail(LM_ERR_INVALID_ARG, "srank_alpha must be > 0");
    if (c->srank_iters < 1 || c->srank_iters > 64) return fail(LM_ERR_INVALID_ARG, "srank_iters must be in [1, 64]");
  }
  const int world = c->shard_world == 0 ? 1 : c->shard_world;
  if (world < 1 || world > 4096) return fail(LM_ERR_INVALID_ARG, "shard_world must be in [0, 4096]");
  if (c->shard_rank < 0 || c->shard_rank >= world)
    return fail(LM_ERR_INVALID_ARG, "shard_rank %d is not in [0, %d)", c->shard_rank, world);
  if (world > 1 && c->schedule != LM_SCHEDULE_PERIOD)
    return fail(LM_ERR_UNSUPPORTED, "layer sharding needs schedule LM_SCHEDULE_PERIOD");
  if (c->vector_rule != LM_VECTOR_LION && c->vector_rule != LM_VECTOR_ADAMW)
    return fail(LM_ERR_INVALID_ARG, "vector_rule must be LM_VECTOR_LION or LM_VECTOR_ADAMW");
  if (c->vector_rule == LM_VECTOR_ADAMW) {
    if (!finite(c->adamw_lr) || c->adamw_lr < 0) return fail(LM_ERR_INVALID_ARG, "adamw_lr must be finite and >= 0");
    if (!(c->adamw_beta1 >= 0.0 && c->adamw_beta1 < 1.0) || !(c->adamw_beta2 >= 0.0 && c->adamw_beta2 < 1.0))
      return fail(LM_ERR_INVALID_ARG, "adamw_beta1/adamw_beta2 must lie in [0, 1)");
    if (!finite(c->adamw_eps) || !(c->adamw_eps > 0)) return fail(LM_ERR_INVALID_ARG, "adamw_eps must be > 0");
    if (!finite(c->adamw_weight_decay) || c->adamw_weight_decay < 0)
      return fail(LM_ERR_INVALID_ARG, "adamw_weight_decay must be >= 0");
  }
  return LM_OK;
}

lm_status check_device(int* dev_out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(LM_ERR_CUDA, "no CUDA device: %s", cudaGetErrorString(e));
  int major = 0, minor = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (major != 10 || minor != 3)
    return fail(LM_ERR_UNSUPPORTED, "device %d is sm_%d%d; this library is built for sm_103a", dev, major, minor);
  *dev_out = dev;
  return LM_OK;
}

LionConsts lion_consts(const lm_config& c) {
  LionConsts k;
  k.b1 = (float)c.beta1;
  k.c1 = (float)(1.0 - c.beta1);
  k.b2 = (float)c.beta2;
  k.c2 = (float)(1.0 - c.beta2);
  k.eL = (float)c.eta_lion;
  k.lam = (float)c.weight_decay;
  k.skip = nullptr;
  k.flags = nullptr;
  return k;
}
// AdamW constants of step t (update number t + 1): powers and the square
// root in double, each constant rounded once to float.
AdamConsts adamw_consts(const lm_config& c, int64_t t) {
  const double k = (double)(t + 1);
  const double bc1 = 1.0 - std::pow(c.adamw_beta1, k);
  const double bc2 = 1.0 - std::pow(c.adamw_beta2, k);
  AdamConsts a;
  a.b1 = (float)c.adamw_beta1;
  a.c1 = (float)(1.0 - c.adamw_beta1);
  a.b2 = (float)c.adamw_beta2;
  a.c2 = (float)(1.0 - c.adamw_beta2);
  a.step = (float)(c.adamw_lr / bc1);
  a.rbc2 = (float)(1.0 / std::sqrt(bc2));
  a.lrwd = (float)(c.adamw_lr * c.adamw_weight_decay);
  a.eps = (float)c.adamw_eps;
  a.flags = nullptr;
  return a;
}

MuonConsts muon_consts(const lm_config& c) {
  MuonConsts k;
  k.b1 = (float)c.beta1;
  k.c1 = (float)(1.0 - c.beta1);
  k.b2 = (float)c.beta2;
  k.c2 = (float)(1.0 - c.beta2);
  k.eM = (float)c.eta_muon;
  k.lam = (float)c.weight_decay;
  k.eps = (float)c.ns_eps;
  k.ns_steps = c.ns_steps;
  k.active = nullptr;
  k.flags = nullptr;
  return k;
}

// Device-memory arena: one cudaMalloc, sub-allocated with 256-byte alignment.
// With guard bands on (LM_DEBUG=1 when the state is created), every part is
// followed by kGuardBytes of a fixed pattern, checked by lm_get_status.
constexpr size_t kGuardBytes = 256;
constexpr unsigned char kGuardByte = 0xA5;
struct Arena {
  std::vector<std::pair<size_t, size_t>> parts;  // (offset, bytes)
  size_t total = 0;
  bool guard = false;
  std::vector<size_t> guards;                     // offsets of the guard bands
  size_t add(size_t bytes) {
    total = align_up(total, 256);
    size_t off = total;
    total += std::max<size_t>(bytes, 1);
    if (guard) {
      total = align_up(total, 256);
      guards.push_back(total);
      total += kGuardBytes;
    }
    return off;
  }
};

// Switches read from the environment when a state is created (or an msign
// call starts; host side only, none of them changes the device code):
//   LM_DEBUG=1         guard bands around every workspace part
//   LM_NVTX=1          NVTX ranges around every kernel family's launches
//   LM_FAULT=oom       lm_create fails with LM_ERR_OOM as if the allocation had
//   LM_NS_FORCE_FP32=1 the fp32 Newton-Schulz path whatever ns_precision says
//   LM_NS_TILES=wide   two-block (256 x 512) Newton-Schulz tiles wherever
//                      they fit, run by the wide-tile kernel; the default
//                      (or LM_NS_TILES=narrow) is one-block tiles.  The
//                      results are the same bit for bit
//   LM_PDL=0           no programmatic dependent launch between NS launches
//   LM_NS_FOLD=0       keep a X as a separate term of APPLY instead of folding
//                      a into B's diagonal
//   LM_WAIT_LIMIT_NS=n limit of every bounded device wait (default 5 s; a
//                      short limit makes waits give up, for failure tests)
static bool env_is(const char* name, const char* value) {
  const char* v = std::getenv(name);
  return v != nullptr && std::strcmp(v, value) == 0;
}
static int env_tiles_mode() {
  if (env_is("LM_NS_TILES", "narrow")) return 1;
  if (env_is("LM_NS_TILES", "wide")) return 2;
  return 0;
}
static std::atomic<bool> g_nvtx{false};
static const char* const kFamilyNames[LM_KERNEL_FAMILIES] = {
    "lion", "momentum_norm", "ns_gram", "ns_poly", "ns_apply", "finalize", "other", "adamw", "srank"};

constexpr int64_t kLionChunk = 32768;   // elements per Lion work chunk
// Three-piece mode: Gram tiles longer than this many 64-deep K blocks (1536)
// are split along K, whatever the balance (the parts are added in fp32): the
// tensor cores' fp32 accumulation error grows with the MMAs summed into one
// accumulator.  Measured on a 720M-set Muon step: the largest direction error
// 2.5e-5 at 96 blocks, 1.2e-5 at 48, 8.8e-6 at 32, 8.4e-6 at 24.
constexpr int kGramCapF32TC = 24;
constexpr uint64_t kRingWaitNs = 2000000000ull;   // the power-iteration ring's waits: 2 s unless set shorter

struct LionTable {
  LionTensor* tensors = nullptr;
  LionChunk* chunks = nullptr;
  int nchunks = 0;
};

// One launch batch of the Newton-Schulz GEMMs: up to kMaxGroupsTc groups
// (tensor-core path) or all groups (fp32 path), a tile list per phase.
struct NsBatch {
  int g0 = 0, ng = 0;
  NsTile* tiles[3] = {nullptr, nullptr, nullptr};
  int ntiles[3] = {0, 0, 0};
  bool wide[3] = {false, false, false};            // tiles of two 256-column blocks: the wide-tile kernel
  int* offsets[3] = {nullptr, nullptr, nullptr};   // per-pair tile ranges (tensor-core path)
  int npairs[3] = {0, 0, 0};
  NsSplitTarget* split_targets = nullptr;   // split Gram tiles of this batch
  int nsplit = 0;
};

struct AdamTable {
  AdamTensor* tensors = nullptr;
  LionChunk* chunks = nullptr;
  int nchunks = 0;
};

template <typename TensorT>
void build_lion_chunks(const std::vector<TensorT>& ts, std::vector<LionChunk>& out) {
  for (size_t i = 0; i < ts.size(); ++i) {
    for (int64_t b = 0; b < ts[i].n; b += kLionChunk) {
      LionChunk c;
      c.tensor = (int32_t)i;
      c.pad = 0;
      c.begin = b;
      c.count = std::min<int64_t>(kLionChunk, ts[i].n - b);
      out.push_back(c);
    }
  }
}

// Tile list of one phase over groups [g0, g0+ng).  Symmetric phases keep the
// tiles that reach the diagonal or above; the list is ordered longest K first.
// Greedy longest-first assignment of tiles (sorted by decreasing cost) to
// workers: each tile goes to the least-loaded worker.  Output: tiles grouped
// by worker and the npairs + 1 range starts.
void balance_tiles(const std::vector<std::pair<int, NsTile>>& sorted, int workers,
                   std::vector<NsTile>& out, std::vector<int>& offsets) {
  std::vector<std::vector<NsTile>> per(workers);
  std::vector<std::pair<int64_t, int>> heap;   // (load, worker), min-heap
  for (int k = 0; k < workers; ++k) heap.push_back({0, k});
  auto cmp = [](const std::pair<int64_t, int>& a, const std::pair<int64_t, int>& b) { return a > b; };
  std::make_heap(heap.begin(), heap.end(), cmp);
  for (const auto& e : sorted) {
    std::pop_heap(heap.begin(), heap.end(), cmp);
    auto& top = heap.back();
    per[top.second].push_back(e.second);
    top.first += e.first;
    std::push_heap(heap.begin(), heap.end(), cmp);
  }
  offsets.assign(1, 0);
  for (int k = 0; k < workers; ++k) {
    out.insert(out.end(), per[k].begin(), per[k].end());
    offsets.push_back((int)out.size());
  }
}

// wide: a tile covers column blocks tn and tn + 1 where both exist (nh = 2).
// APPLY pairs blocks 2k and 2k + 1; the symmetric phases pair the blocks of
// a row from its diagonal block on, (tm, tm + 1), (tm + 2, tm + 3), ..., so
// that every stored block is computed exactly once.
void build_ns_tiles(const std::vector<NsGroup>& groups, int g0, int ng, int phase, int bm, int bn,
                    std::vector<NsTile>& out, bool wide = false) {
  std::vector<std::pair<int, NsTile>> v;
  for (int gi = g0; gi < g0 + ng; ++gi) {
    const NsGroup& g = groups[gi];
    // output rows x cols: s x s (GRAM, POLY), s x l (APPLY wide), l x s (APPLY tall)
    const int nrow = (phase == NS_APPLY && g.tall) ? g.l_pad : g.s_pad;
    const int ncol = (phase == NS_APPLY) ? (g.tall ? g.s_pad : g.l_pad) : g.s_pad;
    const int K = (phase == NS_GRAM) ? g.l_pad : g.s_pad;
    const int tms = (nrow + bm - 1) / bm, tns = (ncol + bn - 1) / bn;
    for (int m = 0; m < g.count; ++m)
      for (int tm = 0; tm < tms; ++tm) {
        int tn = 0;
        if (phase != NS_APPLY)   // first block reaching the diagonal
          while (tn < tns && (int64_t)(tn + 1) * bn <= (int64_t)tm * bm) ++tn;
        while (tn < tns) {
          NsTile t;
          memset(&t, 0, sizeof(t));
          t.group = (uint16_t)(gi - g0);
          t.mat = (uint16_t)m;
          t.tm = (uint16_t)tm;
          t.tn = (uint16_t)tn;
          t.nh = (uint16_t)((wide && tn + 1 < tns) ? 2 : 1);
          v.push_back({K, t});
          tn += t.nh;
        }
      }
  }
  std::stable_sort(v.begin(), v.end(), [](const std::pair<int, NsTile>& a, const std::pair<int, NsTile>& b) {
    return a.first > b.first;
  });
  for (auto& e : v) out.push_back(e.second);
}

// Element chunks of each matrix (kElemChunk elements, the last one ragged).
void build_elem_chunks(const std::vector<MatDesc>& mats, std::vector<ElemChunk>& out) {
  for (size_t i = 0; i < mats.size(); ++i) {
    const int64_t n = mats[i].rows * mats[i].cols;
    for (int64_t b = 0; b < n; b += kElemChunk)
      out.push_back(ElemChunk{(int32_t)i, 0, b, std::min<int64_t>(kElemChunk, n - b)});
  }
}

}  // namespace

lm_status set_error(lm_status st, const char* msg) { return fail(st, "%s", msg); }

// ---------------------------------------------------------------------------
// Newton-Schulz engine shared by lm_step and lm_msign_ns
// ---------------------------------------------------------------------------
struct NsEngine {
  lm_dtype xdt = LM_BF16;            // workspace dtype: bf16 (tensor cores) or fp32
  int pieces = 1;                    // tensor cores: 3 = fp32 values as three bf16 planes
  std::vector<NsGroup> groups;       // host copies (device pointers inside)
  std::vector<TcGroupMaps> maps;     // tensor-core path
  NsGroup* d_groups = nullptr;       // fp32 path reads groups from device memory
  std::vector<NsBatch> batches;
  double* d_norm2 = nullptr;
  float* d_split_ws = nullptr;       // fp32 partial sums of split Gram tiles
  bool pdl = true;                   // programmatic dependent launch between NS launches
  bool fold = true;                  // fold a into B's diagonal where |a| < 4 (bf16 operands)
  uint64_t wait_ns = kDefaultWaitNs; // limit of the kernels' bounded waits
};

// Plan: group matrices by (s, l); returns matrix order (indices into shapes)
// and fills groups with sizes (pointers set later).
static void plan_groups(const std::vector<std::pair<int64_t, int64_t>>& shapes, lm_dtype xdt,
                        std::vector<NsGroup>& groups, std::vector<std::vector<int>>& members) {
  // one group per (rows, cols): same (s, l) but opposite orientation are
  // different groups, since X keeps the parameter's orientation
  std::map<std::pair<int64_t, int64_t>, int> key_to_group;
  for (size_t i = 0; i < shapes.size(); ++i) {
    const int64_t s = std::min(shapes[i].first, shapes[i].second);
    const int64_t l = std::max(shapes[i].first, shapes[i].second);
    auto key = shapes[i];
    auto it = key_to_group.find(key);
    if (it == key_to_group.end()) {
      NsGroup g;
      memset(&g, 0, sizeof(g));
      g.s = (int32_t)s;
      g.l = (int32_t)l;
      g.tall = shapes[i].first > shapes[i].second ? 1 : 0;
      if (xdt == LM_BF16) {
        g.s_pad = tc_pad_s((int)s);
        g.l_pad = tc_pad_l((int)l);
      } else {
        g.s_pad = simt_pad((int)s);
        g.l_pad = simt_pad((int)l);
      }
      key_to_group[key] = (int)groups.size();
      groups.push_back(g);
      members.emplace_back();
      it = key_to_group.find(key);
    }
    members[it->second].push_back((int)i);
  }
  int first = 0;
  for (size_t gi = 0; gi < groups.size(); ++gi) {
    groups[gi].count = (int32_t)members[gi].size();
    groups[gi].first_mat = first;
    first += groups[gi].count;
  }
}

// Reserve workspace for the groups and the tile lists in the arena.
struct NsLayout {
  std::vector<size_t> off_x0, off_x1, off_a, off_b, off_xf;
  std::vector<std::vector<NsTile>> tiles;   // per batch*3 + phase
  std::vector<size_t> off_tiles;
  std::vector<std::vector<int>> offsets;    // per batch*3 + phase (tensor-core path)
  std::vector<size_t> off_offsets;
  size_t off_groups = 0;
  size_t off_norm = 0;
  // split Gram tiles, per batch: (group, mat, tm, tn, first part, parts) of each target tile
  std::vector<std::vector<std::array<int, 6>>> split_targets;
  std::vector<size_t> off_split_targets;
  size_t off_split_ws = 0;
};

// Split-K of the Gram phase: a tile longer than twice the average load of a
// worker (a CTA pair on the tensor-core path, a block on the fp32 path) - a
// long-K embedding Gram next to short hidden matrices, which would otherwise
// set the length of the launch - is cut into parts of at most half that load.
// Each part is a tile of its own for the scheduler and writes its partial
// product to a workspace tile of its own (slot = part index + 1); the finish
// kernel adds the parts in order, so the result does not depend on timing.
// Tiles near the average stay whole: splitting them buys no balance.
// kcap > 0 also splits every tile longer than kcap K slices into parts of at
// most kcap: the three-piece fp32 mode bounds the length of each fp32
// accumulation in TMEM that way (the parts are added in fp32 by the finish
// kernel).
static void split_gram_tiles(const std::vector<NsGroup>& groups, int g0, std::vector<NsTile>& t, int kslice,
                             int workers, std::vector<std::array<int, 6>>& targets, int& nparts_total,
                             int kcap = 0) {
  int64_t total = 0;
  for (const NsTile& x : t) total += (int64_t)(groups[g0 + x.group].l_pad / kslice) * (x.nh == 2 ? 2 : 1);
  const int64_t avg = total / std::max(1, workers);
  int64_t part = std::max<int64_t>(8, avg / 2);
  if (kcap > 0) part = std::min<int64_t>(part, kcap);
  std::vector<NsTile> out;
  nparts_total = 0;
  for (const NsTile& x0 : t) {
    const int nk = groups[g0 + x0.group].l_pad / kslice;
    const int nh = x0.nh == 2 ? 2 : 1;
    // decided per 256-column block, so that one- and two-block tiles split
    // the same blocks into the same parts (and give the same sums)
    if ((nk <= 2 * avg && (kcap <= 0 || nk <= kcap)) || nparts_total + 128 > 65535) {
      out.push_back(x0);
      continue;
    }
    // a split tile is one block wide: a two-block tile is split per block
    for (int h = 0; h < nh; ++h) {
      NsTile x = x0;
      x.tn = (uint16_t)(x0.tn + h);
      x.nh = 1;
      const int nparts = (int)std::min<int64_t>(64, (nk + part - 1) / part);
      targets.push_back({x.group, x.mat, x.tm, x.tn, nparts_total, nparts});
      for (int k = 0; k < nparts; ++k) {
        NsTile y = x;
        y.kb0 = (uint16_t)((int64_t)nk * k / nparts);
        y.kb1 = (uint16_t)((int64_t)nk * (k + 1) / nparts);
        y.slot = (uint16_t)(nparts_total + k + 1);
        out.push_back(y);
      }
      nparts_total += nparts;
    }
  }
  t.swap(out);
}

// tiles_mode: 0 or 1 one-block tiles, 2 two-block tiles wherever a row has
// two blocks left (bf16 operands).
static void layout_ns(std::vector<NsGroup>& groups, lm_dtype xdt, int nmat, Arena& ar, NsLayout& L,
                      std::vector<NsBatch>& batches, int pieces = 1, int tiles_mode = 0) {
  const size_t es = dtype_size(xdt) * (size_t)pieces;
  for (auto& g : groups) {
    const size_t xb = (size_t)g.count * g.s_pad * g.l_pad * es;
    const size_t ab = (size_t)g.count * g.s_pad * g.s_pad * es;
    L.off_x0.push_back(ar.add(xb));
    L.off_x1.push_back(ar.add(xb));
    L.off_a.push_back(ar.add(ab));
    L.off_b.push_back(ar.add(ab));
    // three-piece mode: fp32 X_0 / X_K
    L.off_xf.push_back(pieces == 3 ? ar.add((size_t)g.count * g.s_pad * g.l_pad * sizeof(float)) : 0);
  }
  const int per = (xdt == LM_BF16) ? kMaxGroupsTc : kMaxGroupsSimt;
  int max_split = 0;
  const int bm = (xdt == LM_BF16) ? kTcBM : kSimtBM;
  const int bn = (xdt == LM_BF16) ? kTcBN : kSimtBN;
  for (int g0 = 0; g0 < (int)groups.size(); g0 += per) {
    NsBatch b;
    b.g0 = g0;
    b.ng = std::min(per, (int)groups.size() - g0);
    for (int ph = 0; ph < 3; ++ph) {
      std::vector<NsTile> t;
      build_ns_tiles(groups, g0, b.ng, ph, bm, bn, t);
      // Two-block tiles stage a quarter fewer bytes per FLOP, but they take
      // both accumulators (the epilogue of one tile no longer overlaps the
      // next tile's main loop), leave room for a 3- or 4-stage ring only and
      // put twice as many matrices in flight in a launch (a larger L2 working
      // set): measured slower on the GPT-style sets, so used only on request.
      if (xdt == LM_BF16 && pieces == 1 && tiles_mode == 2) {
        t.clear();
        build_ns_tiles(groups, g0, b.ng, ph, bm, bn, t, true);
        b.wide[ph] = true;
      }
      std::vector<int> offs;
      std::vector<std::array<int, 6>> targets;
      if (ph == NS_GRAM) {
        int nparts = 0;
        if (xdt == LM_BF16) {
          // three-piece mode: no fp32 accumulation over more than kGramCapF32TC K blocks
          split_gram_tiles(groups, g0, t, kTcBK, tc_max_pairs(), targets, nparts, pieces == 3 ? kGramCapF32TC : 0);
        } else {
          int dev = 0, sms = 0;
          cudaGetDevice(&dev);
          cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
          split_gram_tiles(groups, g0, t, 16, 2 * std::max(sms, 1), targets, nparts);
        }
        b.nsplit = (int)targets.size();
        max_split = std::max(max_split, nparts);
        L.off_split_targets.push_back(ar.add(targets.size() * sizeof(NsSplitTarget)));
        L.split_targets.push_back(std::move(targets));
      }
      if (xdt == LM_BF16 && !t.empty()) {
        // cost of a tile: its K blocks plus an allowance for the epilogue
        std::vector<std::pair<int, NsTile>> sorted;
        for (const NsTile& x : t) {
          const NsGroup& g = groups[g0 + x.group];
          const int nk = (ph == NS_GRAM) ? (x.kb1 != 0 ? x.kb1 - x.kb0 : g.l_pad / kTcBK) : g.s_pad / kTcBK;
          sorted.push_back({(nk + 6) * (x.nh == 2 ? 2 : 1), x});
        }
        std::stable_sort(sorted.begin(), sorted.end(),
                         [](const std::pair<int, NsTile>& a, const std::pair<int, NsTile>& c) {
                           return a.first > c.first;
                         });
        const int workers = std::min<int>(tc_max_pairs(), (int)t.size());
        t.clear();
        balance_tiles(sorted, workers, t, offs);
        b.npairs[ph] = workers;
      }
      b.ntiles[ph] = (int)t.size();
      L.off_tiles.push_back(ar.add(t.size() * sizeof(NsTile)));
      L.tiles.push_back(std::move(t));
      L.off_offsets.push_back(ar.add(offs.size() * sizeof(int)));
      L.offsets.push_back(std::move(offs));
    }
    batches.push_back(b);
  }
  L.off_groups = ar.add(groups.size() * sizeof(NsGroup));
  L.off_norm = ar.add((size_t)std::max(nmat, 1) * sizeof(double));
  const size_t tile_floats = (xdt == LM_BF16) ? (size_t)kTcBM * kTcBN : (size_t)kSimtBM * kSimtBN;
  L.off_split_ws = ar.add((size_t)max_split * tile_floats * sizeof(float));
}

static void bind_ns(NsEngine& E, char* base, const NsLayout& L, std::vector<char>& host_img) {
  for (size_t gi = 0; gi < E.groups.size(); ++gi) {
    E.groups[gi].X[0] = base + L.off_x0[gi];
    E.groups[gi].X[1] = base + L.off_x1[gi];
    E.groups[gi].A = base + L.off_a[gi];
    E.groups[gi].B = base + L.off_b[gi];
    E.groups[gi].Xf = E.pieces == 3 ? base + L.off_xf[gi] : nullptr;
  }
  for (size_t bi = 0; bi < E.batches.size(); ++bi)
    for (int ph = 0; ph < 3; ++ph) {
      const size_t k = bi * 3 + ph;
      E.batches[bi].tiles[ph] = reinterpret_cast<NsTile*>(base + L.off_tiles[k]);
      if (!L.tiles[k].empty())
        memcpy(host_img.data() + L.off_tiles[k], L.tiles[k].data(), L.tiles[k].size() * sizeof(NsTile));
      if (!L.offsets[k].empty()) {
        E.batches[bi].offsets[ph] = reinterpret_cast<int*>(base + L.off_offsets[k]);
        memcpy(host_img.data() + L.off_offsets[k], L.offsets[k].data(), L.offsets[k].size() * sizeof(int));
      }
    }
  for (size_t bi = 0; bi < E.batches.size(); ++bi) {
    const auto& tg = L.split_targets[bi];
    std::vector<NsSplitTarget> st(tg.size());
    const bool tc = E.xdt == LM_BF16;
    const size_t es = tc ? 2 : 4;                 // A: bf16 (tensor cores) or fp32
    const int tile = tc ? kTcBM : kSimtBM;
    for (size_t k = 0; k < tg.size(); ++k) {
      const NsGroup& g = E.groups[E.batches[bi].g0 + tg[k][0]];
      char* a = static_cast<char*>(g.A) + (size_t)tg[k][1] * g.s_pad * g.s_pad * es;
      const int tm = tg[k][2], tn = tg[k][3];
      st[k].a_tile = a + ((size_t)tm * tile * g.s_pad + (size_t)tn * tile) * es;
      st[k].a_mirror = a + ((size_t)tn * tile * g.s_pad + (size_t)tm * tile) * es;
      st[k].ld = g.s_pad;
      st[k].nr = std::min(tile, g.s_pad - tm * tile);
      st[k].nc = std::min(tile, g.s_pad - tn * tile);
      st[k].first = tg[k][4];
      st[k].nparts = tg[k][5];
      st[k].diag = tm == tn ? 1 : 0;
      st[k].plane = (tc && E.pieces == 3) ? (int64_t)g.count * g.s_pad * g.s_pad : 0;
    }
    E.batches[bi].split_targets = reinterpret_cast<NsSplitTarget*>(base + L.off_split_targets[bi]);
    if (!st.empty()) memcpy(host_img.data() + L.off_split_targets[bi], st.data(), st.size() * sizeof(NsSplitTarget));
  }
  E.d_split_ws = reinterpret_cast<float*>(base + L.off_split_ws);
  E.d_groups = reinterpret_cast<NsGroup*>(base + L.off_groups);
  memcpy(host_img.data() + L.off_groups, E.groups.data(), E.groups.size() * sizeof(NsGroup));
  E.d_norm2 = reinterpret_cast<double*>(base + L.off_norm);
}

static lm_status encode_maps(NsEngine& E) {
  if (E.xdt != LM_BF16) return LM_OK;
  E.maps.resize(E.groups.size());
  for (size_t gi = 0; gi < E.groups.size(); ++gi) {
    cudaError_t e = tc_encode_group_maps(E.groups[gi], &E.maps[gi], E.pieces);
    if (e != cudaSuccess) return cuda_fail(e, "cuTensorMapEncodeTiled");
  }
  return LM_OK;
}

// Event timing of kernel launches (enabled by lm_profile_enable).
struct Profiler {
  bool on = false;
  struct Rec {
    int fam;
    cudaEvent_t a, b;
  };
  std::vector<cudaEvent_t> pool;
  size_t used = 0;
  std::vector<Rec> recs;
  double ms[LM_KERNEL_FAMILIES] = {0};
  uint64_t n[LM_KERNEL_FAMILIES] = {0};
  cudaEvent_t next() {
    if (used == pool.size()) {
      cudaEvent_t e = nullptr;
      if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
      pool.push_back(e);
    }
    return pool[used++];
  }
  ~Profiler() {
    for (cudaEvent_t e : pool) cudaEventDestroy(e);
  }
};

// Launch f() on st; with profiling on, bracket it by events of family fam.
template <typename F>
static cudaError_t timed_events(Profiler* P, int fam, cudaStream_t st, F&& f) {
  if (P == nullptr || !P->on) return f();
  // launches being captured into a graph are not timed (their events would
  // be graph nodes, not measurements)
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (st != nullptr && cudaStreamIsCapturing(st, &cap) == cudaSuccess && cap != cudaStreamCaptureStatusNone)
    return f();
  cudaEvent_t a = P->next(), b = P->next();
  if (a == nullptr || b == nullptr) return f();
  cudaEventRecord(a, st);
  cudaError_t e = f();
  cudaEventRecord(b, st);
  P->recs.push_back({fam, a, b});
  return e;
}

// timed_events plus an NVTX range named after the family when LM_NVTX=1.
template <typename F>
static cudaError_t timed(Profiler* P, int fam, cudaStream_t st, F&& f) {
  const bool nvtx = g_nvtx.load(std::memory_order_relaxed);
  if (nvtx) nvtxRangePushA(kFamilyNames[fam]);
  cudaError_t e = timed_events(P, fam, st, std::forward<F>(f));
  if (nvtx) nvtxRangePop();
  return e;
}

// Per-iteration coefficients: (a_k, b_k, c_k) from a 3 * steps table, or the
// constant (a, b, c) when the table is NULL; eps goes with every iteration.
static std::vector<NsCoeffs> ns_schedule(int steps, const double* table, double a, double b, double c,
                                         double eps) {
  std::vector<NsCoeffs> co((size_t)std::max(steps, 0));
  for (int k = 0; k < steps; ++k) {
    const double* t = table ? table + 3 * k : nullptr;
    co[k] = NsCoeffs{(float)(t ? t[0] : a), (float)(t ? t[1] : b), (float)(t ? t[2] : c), (float)eps};
  }
  return co;
}

static lm_status run_ns(const NsEngine& E, int steps, const NsCoeffs* coeffs, unsigned* flags, cudaStream_t st,
                        Profiler* P = nullptr, const FuseFinal* fuse = nullptr,
                        const unsigned char* active = nullptr) {
  // three-piece mode: X_0 (fp32, from the momentum kernel) -> bf16 planes
  for (size_t gi = 0; E.pieces == 3 && steps > 0 && gi < E.groups.size(); ++gi) {
    const NsGroup& g = E.groups[gi];
    cudaError_t e = timed(P, LM_KERNEL_OTHER, st, [&]() {
      return launch_split3(static_cast<const float*>(g.Xf), g.X[0], (size_t)g.count * g.s_pad * g.l_pad, flags, st);
    });
    if (e != cudaSuccess) return cuda_fail(e, "three-piece split launch");
  }
  for (int it = 0; it < steps; ++it)
    for (const NsBatch& b : E.batches)
      for (int ph = 0; ph < 3; ++ph) {
        const NsCoeffs co = coeffs[it];
        // an iteration without the A^2 term (c = 0, a cubic): B = b A is not
        // formed; the tensor-core APPLY reads A and scales by b instead
        const bool from_a = E.xdt == LM_BF16 && co.c == 0.f && !b.wide[NS_POLY] && !b.wide[NS_APPLY];
        if (ph == NS_POLY && from_a) continue;
        // an iteration whose |a| is below 4: POLY stores B' = a I + B and APPLY
        // computes X' = B' X with no X tile in its epilogue (bf16 operands,
        // one-block tiles).  On the constant quintic this also lowers the
        // error against the fp64 iteration (bf16 msign: 6.2e-3 against 8.3e-3
        // on 1280 x 5120, 6.5e-3 against 1.0e-2 on 768 x 50304); a larger a
        // (the first minimax iterations, 8.47) would round the diagonal too
        // coarsely.
        const bool fold = E.fold && E.xdt == LM_BF16 && E.pieces == 1 && !from_a && std::fabs(co.a) < 4.f &&
                          !b.wide[NS_POLY] && !b.wide[NS_APPLY];
        const bool split = E.xdt == LM_BF16 && ph == NS_GRAM && b.nsplit > 0;
        cudaError_t e = timed(P, LM_KERNEL_NS_GRAM + ph, st, [&]() {
          if (E.xdt == LM_BF16) {
            cudaError_t r = launch_ns_tc((NsPhase)ph, it, b.ng, E.groups.data() + b.g0, E.maps.data() + b.g0, b.tiles[ph],
                               b.ntiles[ph], b.offsets[ph], b.npairs[ph], E.d_norm2, co, flags,
                               it == steps - 1 ? fuse : nullptr, st, active, split ? E.d_split_ws : nullptr,
                               E.pieces, it == steps - 1 ? 1 : 0, b.wide[ph], E.pdl, E.wait_ns,
                               ph == NS_APPLY && from_a, ph != NS_GRAM && fold);
            if (r == cudaSuccess && split)
              r = launch_ns_split_finish(b.split_targets, b.nsplit, E.d_split_ws, flags, st);
            return r;
          }
          cudaError_t r = launch_ns_simt((NsPhase)ph, it, b.ng, E.d_groups + b.g0, b.tiles[ph], b.ntiles[ph],
                                         E.d_norm2, co, st, active, E.d_split_ws, flags);
          if (r == cudaSuccess && ph == NS_GRAM && b.nsplit > 0)
            r = launch_ns_split_finish_f32(b.split_targets, b.nsplit, E.d_split_ws, flags, st);
          return r;
        });
        if (e != cudaSuccess) return cuda_fail(e, "Newton-Schulz launch");
      }
  return LM_OK;
}

}  // namespace lm

using namespace lm;

// Layer sharding (Section 5.4): whole matrices dealt out to `world` ranks,
// largest Newton-Schulz cost 3 s^2 l + s^3 first, each to the least-loaded
// rank (the lowest on a tie); ties in cost keep parameter order.  1-D
// parameters: -1.
static void shard_owners(const lm_tensor* params, int n, int world, std::vector<int>& owner) {
  owner.assign(n, -1);
  std::vector<std::pair<double, int>> cost;
  for (int i = 0; i < n; ++i)
    if (is_matrix(params[i])) {
      const double s = (double)std::min(params[i].rows, params[i].cols);
      const double l = (double)std::max(params[i].rows, params[i].cols);
      cost.push_back({3.0 * s * s * l + s * s * s, i});
    }
  std::stable_sort(cost.begin(), cost.end(),
                   [](const std::pair<double, int>& a, const std::pair<double, int>& b) { return a.first > b.first; });
  std::vector<double> load(std::max(world, 1), 0.0);
  for (const auto& c : cost) {
    const int r = (int)(std::min_element(load.begin(), load.end()) - load.begin());
    owner[c.second] = r;
    load[r] += c.first;
  }
}

// ---------------------------------------------------------------------------
// the state
// ---------------------------------------------------------------------------
struct lm_state {
  int device = 0;
  lm_config cfg;
  int n = 0;
  std::vector<lm_tensor> params;
  std::vector<size_t> mom_off;      // element offset of each momentum buffer
  size_t mom_elems = 0;             // sum |W_i|
  char* base = nullptr;             // the one device allocation
  size_t bytes = 0;
  float* mom = nullptr;
  const void** d_grads = nullptr;   // device grad-pointer table
  std::vector<const void*> h_grads; // what the device table holds
  std::vector<const void*> grads_checked;   // gradient pointers found to be device memory
  bool grads_valid = false;
  LionTable lion_all[2], lion_vec[2];   // lion_all: matrices only under LM_VECTOR_ADAMW
  int world = 1, rank = 0;              // layer sharding: this state's rank of `world`
  std::vector<int> owner;               // owner rank per parameter (-1: 1-D), sharded states
  LionTable ema[2];                     // matrices other ranks own: momentum update on Muon steps
  bool adamw = false;                   // 1-D parameters take AdamW
  AdamTable adam[2];                    // per dtype, 1-D parameters
  float* vmom = nullptr;                // AdamW second moments
  std::vector<int64_t> v_off;           // element offset per parameter, -1 if none
  size_t v_elems = 0;
  // stable-rank selection (LM_SCHEDULE_STABLE_RANK)
  struct SrLaunch {
    int slots = 0, threads = 0;
    bool vec4 = false;                  // rows are 16-byte multiples: the ring kernel
    int64_t max_cols = 0;
    SrItem* items = nullptr;
    int nitems = 0;
  };
  bool srank = false;
  SrMat* d_sr = nullptr;                // per matrix id
  std::vector<SrLaunch> sr_launch;
  float* sr_wa = nullptr;
  float* sr_wb = nullptr;
  size_t sr_w_elems = 0;                // floats in each of wa, wb
  double* sr_acc = nullptr;             // nmat x (1 + srank_iters)
  unsigned char* d_active = nullptr;    // per matrix id: takes Muon this step
  unsigned char* d_skip = nullptr;      // per parameter: Lion kernel skips it
  double* d_srank = nullptr;            // per matrix id: the estimate
  std::vector<int> mat_param_of;        // matrix id -> parameter index
  // With two or more column-count launches per pass, launches after the
  // first go to side streams forked from and joined back to the caller's
  // stream, so that one launch's last blocks overlap the next launch.
  cudaStream_t sr_side[2] = {nullptr, nullptr};
  cudaEvent_t sr_fork = nullptr, sr_join[2] = {nullptr, nullptr};
  int sr_nside = 0;
  int64_t last_t = -1;
  // LM_DEBUG guard bands: device list of their offsets
  bool debug = false;
  size_t* d_guard_offs = nullptr;
  int n_guards = 0;
  int lion_grid[2] = {0, 0};
  int nmat = 0;
  MatDesc* d_mats = nullptr;
  bool fuse_final = false;   // parameter write in the last APPLY epilogue
  CUtensorMap* d_wmaps = nullptr;   // TMA maps of every matrix's W (two each) for that write
  ElemChunk* d_echunks[2] = {nullptr, nullptr};   // chunks of bf16 / fp32 matrices
  int n_echunks[2] = {0, 0};
  NsEngine ns;
  std::vector<NsCoeffs> ns_co;      // coefficients of each NS iteration
  unsigned* d_flags = nullptr;
  cudaStream_t last_stream = nullptr;
  bool captured = false;             // a step of this state was captured into a graph
  Profiler prof;
};

// Side streams of the stable-rank passes (non-blocking, device of lm_create)
// and the events that fork them from and join them to the caller's stream.
static cudaError_t create_side_streams(lm_state* s) {
  s->sr_nside = std::min<int>(2, (int)s->sr_launch.size() - 1);
  cudaError_t e = cudaEventCreateWithFlags(&s->sr_fork, cudaEventDisableTiming);
  for (int k = 0; e == cudaSuccess && k < s->sr_nside; ++k) {
    e = cudaStreamCreateWithFlags(&s->sr_side[k], cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&s->sr_join[k], cudaEventDisableTiming);
  }
  return e;
}

static void destroy_side_streams(lm_state* s) {
  for (int k = 0; k < 2; ++k) {
    if (s->sr_join[k]) cudaEventDestroy(s->sr_join[k]);
    if (s->sr_side[k]) cudaStreamDestroy(s->sr_side[k]);
    s->sr_join[k] = nullptr;
    s->sr_side[k] = nullptr;
  }
  if (s->sr_fork) cudaEventDestroy(s->sr_fork);
  s->sr_fork = nullptr;
  s->sr_nside = 0;
}

extern "C" {

void lm_config_default(lm_config* c) {
  if (c == nullptr) return;
  c->beta1 = 0.9;
  c->beta2 = 0.99;
  c->eta_muon = 3e-3;
  c->eta_lion = 2e-5;
  c->weight_decay = 0.1;
  c->period = 2;
  c->ns_steps = 5;
  c->ns_a = 3.4445;
  c->ns_b = -4.7750;
  c->ns_c = 2.0315;
  c->ns_eps = 1e-7;
  c->shape_scale = 0.2;
  c->ns_precision = LM_BF16;
  c->ns_coeffs = nullptr;
  c->vector_rule = LM_VECTOR_LION;
  c->adamw_lr = 1e-3;
  c->adamw_beta1 = 0.8;
  c->adamw_beta2 = 0.999;
  c->adamw_eps = 1e-8;
  c->adamw_weight_decay = 0.1;
  c->schedule = LM_SCHEDULE_PERIOD;
  c->srank_alpha = 0.01;
  c->srank_iters = 5;
  c->srank_seed = 0;
  c->shard_rank = 0;
  c->shard_world = 1;
}

size_t lm_config_size(void) { return sizeof(lm_config); }

const char* lm_status_string(lm_status st) {
  switch (st) {
    case LM_OK: return "LM_OK";
    case LM_ERR_INVALID_ARG: return "LM_ERR_INVALID_ARG";
    case LM_ERR_DTYPE: return "LM_ERR_DTYPE";
    case LM_ERR_ALIGN: return "LM_ERR_ALIGN";
    case LM_ERR_OOM: return "LM_ERR_OOM";
    case LM_ERR_CUDA: return "LM_ERR_CUDA";
    case LM_ERR_UNSUPPORTED: return "LM_ERR_UNSUPPORTED";
    case LM_ERR_TIMEOUT: return "LM_ERR_TIMEOUT";
  }
  return "unknown lm_status";
}

const char* lm_last_error(void) { return g_last_error.c_str(); }

uint64_t lm_kernel_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

lm_status lm_shard_owners(const lm_tensor* params, int n, int world, int* owner) {
  if (params == nullptr || owner == nullptr) return fail(LM_ERR_INVALID_ARG, "params/owner is NULL");
  if (n < 1) return fail(LM_ERR_INVALID_ARG, "n must be >= 1");
  if (world < 1 || world > 4096) return fail(LM_ERR_INVALID_ARG, "world must be in [1, 4096]");
  for (int i = 0; i < n; ++i)
    if (params[i].rows < 0 || params[i].cols < 0) return fail(LM_ERR_INVALID_ARG, "params[%d] has a negative size", i);
  std::vector<int> o;
  shard_owners(params, n, world, o);
  std::copy(o.begin(), o.end(), owner);
  return LM_OK;
}

lm_status lm_create(const lm_tensor* params, int n, const lm_config* cfg, void* cuda_stream,
                    lm_state** out) {
  if (out == nullptr) return fail(LM_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (params == nullptr || cfg == nullptr) return fail(LM_ERR_INVALID_ARG, "params/cfg is NULL");
  if (n < 1) return fail(LM_ERR_INVALID_ARG, "n must be >= 1");
  lm_status st = check_config(cfg);
  if (st != LM_OK) return st;
  for (int i = 0; i < n; ++i)
    if ((st = check_tensor(&params[i], "params", i)) != LM_OK) return st;
  int dev = 0;
  if ((st = check_device(&dev)) != LM_OK) return st;
  for (int i = 0; i < n; ++i)
    if ((st = check_device_memory(&params[i], "params", i, dev)) != LM_OK) return st;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);

  lm_state* s = new lm_state();
  s->device = dev;
  s->cfg = *cfg;
  s->ns_co = ns_schedule(cfg->ns_steps, cfg->ns_coeffs, cfg->ns_a, cfg->ns_b, cfg->ns_c, cfg->ns_eps);
  s->cfg.ns_coeffs = nullptr;   // the caller's table is not kept
  s->n = n;
  s->params.assign(params, params + n);
  s->ns.xdt = (cfg->ns_precision == LM_F32 || env_is("LM_NS_FORCE_FP32", "1")) ? LM_F32 : LM_BF16;
  s->ns.pieces = (s->ns.xdt == LM_BF16 && cfg->ns_precision == LM_NS_F32_TC) ? 3 : 1;
  s->debug = env_is("LM_DEBUG", "1");
  if (env_is("LM_NVTX", "1")) g_nvtx.store(true);

  // matrices and their shape groups (under layer sharding: the matrices this
  // rank owns; the others only take the momentum update on Muon steps)
  s->world = cfg->shard_world > 1 ? cfg->shard_world : 1;
  s->rank = s->world > 1 ? cfg->shard_rank : 0;
  if (s->world > 1) shard_owners(params, n, s->world, s->owner);
  auto owned = [&](int i) { return s->world == 1 || s->owner[i] == s->rank; };
  std::vector<int> mat_param;
  std::vector<std::pair<int64_t, int64_t>> mat_shapes;
  for (int i = 0; i < n; ++i)
    if (is_matrix(params[i]) && owned(i)) {
      mat_param.push_back(i);
      mat_shapes.push_back({params[i].rows, params[i].cols});
    }
  std::vector<std::vector<int>> members;
  plan_groups(mat_shapes, s->ns.xdt, s->ns.groups, members);
  s->nmat = (int)mat_param.size();

  // arena layout
  Arena ar;
  ar.guard = s->debug;
  s->mom_off.resize(n);
  size_t mom_elems_aligned = 0;
  for (int i = 0; i < n; ++i) {
    s->mom_off[i] = mom_elems_aligned;
    mom_elems_aligned = align_up(mom_elems_aligned + (size_t)numel(params[i]), 64);
    s->mom_elems += (size_t)numel(params[i]);
  }
  const size_t off_mom = ar.add(mom_elems_aligned * sizeof(float));
  // AdamW second moments of the 1-D parameters
  s->adamw = cfg->vector_rule == LM_VECTOR_ADAMW;
  s->v_off.assign(n, -1);
  size_t v_aligned = 0;
  if (s->adamw)
    for (int i = 0; i < n; ++i)
      if (!is_matrix(params[i])) {
        s->v_off[i] = (int64_t)v_aligned;
        v_aligned = align_up(v_aligned + (size_t)numel(params[i]), 64);
        s->v_elems += (size_t)numel(params[i]);
      }
  const size_t off_v = ar.add(v_aligned * sizeof(float));
  const size_t off_grads = ar.add((size_t)n * sizeof(void*));
  const size_t off_flags = ar.add(sizeof(unsigned));

  // Lion tables (per dtype): all params, and vectors only
  std::vector<LionTensor> lt_all[2], lt_vec[2];
  for (int i = 0; i < n; ++i) {
    if (numel(params[i]) == 0) continue;
    LionTensor t;
    t.w = params[i].data;
    t.m = nullptr;   // bound after allocation
    t.n = numel(params[i]);
    t.grad_slot = i;
    t.pad = i;       // remember the param index until binding
    if (!s->adamw || is_matrix(params[i])) lt_all[params[i].dtype].push_back(t);
    if (!is_matrix(params[i])) lt_vec[params[i].dtype].push_back(t);
  }
  // AdamW tables (per dtype) over the 1-D parameters
  std::vector<AdamTensor> at[2];
  std::vector<LionChunk> ac[2];
  size_t off_at[2], off_ac[2];
  for (int i = 0; s->adamw && i < n; ++i) {
    if (numel(params[i]) == 0 || is_matrix(params[i])) continue;
    AdamTensor t;
    t.w = params[i].data;
    t.m = nullptr;
    t.v = nullptr;
    t.n = numel(params[i]);
    t.grad_slot = i;
    t.pad = i;
    at[params[i].dtype].push_back(t);
  }
  for (int d = 0; d < 2; ++d) {
    build_lion_chunks(at[d], ac[d]);
    off_at[d] = ar.add(at[d].size() * sizeof(AdamTensor));
    off_ac[d] = ar.add(ac[d].size() * sizeof(LionChunk));
  }
  // momentum-only table: matrices another rank owns (layer sharding)
  std::vector<LionTensor> lt_ema[2];
  for (int i = 0; i < n; ++i) {
    if (numel(params[i]) == 0 || !is_matrix(params[i]) || owned(i)) continue;
    LionTensor t;
    t.w = params[i].data;
    t.m = nullptr;
    t.n = numel(params[i]);
    t.grad_slot = i;
    t.pad = i;
    lt_ema[params[i].dtype].push_back(t);
  }
  std::vector<LionChunk> lc_all[2], lc_vec[2], lc_ema[2];
  size_t off_lt_all[2], off_lc_all[2], off_lt_vec[2], off_lc_vec[2], off_lt_ema[2], off_lc_ema[2];
  for (int d = 0; d < 2; ++d) {
    build_lion_chunks(lt_all[d], lc_all[d]);
    build_lion_chunks(lt_vec[d], lc_vec[d]);
    build_lion_chunks(lt_ema[d], lc_ema[d]);
    off_lt_all[d] = ar.add(lt_all[d].size() * sizeof(LionTensor));
    off_lc_all[d] = ar.add(lc_all[d].size() * sizeof(LionChunk));
    off_lt_vec[d] = ar.add(lt_vec[d].size() * sizeof(LionTensor));
    off_lc_vec[d] = ar.add(lc_vec[d].size() * sizeof(LionChunk));
    off_lt_ema[d] = ar.add(lt_ema[d].size() * sizeof(LionTensor));
    off_lc_ema[d] = ar.add(lc_ema[d].size() * sizeof(LionChunk));
  }

  // Muon tables
  NsLayout L;
  layout_ns(s->ns.groups, s->ns.xdt, s->nmat, ar, L, s->ns.batches, s->ns.pieces, env_tiles_mode());
  s->ns.pdl = !env_is("LM_PDL", "0");
  s->ns.fold = !env_is("LM_NS_FOLD", "0");
  s->ns.wait_ns = env_wait_limit_ns();
  const size_t off_mats = ar.add((size_t)std::max(s->nmat, 1) * sizeof(MatDesc));
  // TMA maps of W for the parameter write in the last APPLY (bf16 tensor-core path)
  const bool want_wmaps = s->ns.xdt == LM_BF16 && s->ns.pieces == 1 && s->nmat > 0;
  const size_t off_wmaps = want_wmaps ? ar.add((size_t)s->nmat * 2 * sizeof(CUtensorMap)) : 0;
  std::vector<MatDesc> mats(s->nmat);
  // matrices are numbered in group order
  std::vector<int> mat_order;   // mat id -> index into mat_param
  for (size_t gi = 0; gi < members.size(); ++gi)
    for (int m : members[gi]) mat_order.push_back(m);
  for (int id = 0; id < s->nmat; ++id) {
    const lm_tensor& p = params[mat_param[mat_order[id]]];
    MatDesc& d = mats[id];
    memset(&d, 0, sizeof(d));
    d.rows = p.rows;
    d.cols = p.cols;
  }
  // element chunks, split by the parameter dtype (filled once dtypes are bound)
  std::vector<ElemChunk> echunks_all;
  build_elem_chunks(mats, echunks_all);
  const size_t off_echunks = ar.add(echunks_all.size() * sizeof(ElemChunk));

  // stable-rank selection: vectors v0 / wa / wb per matrix, accumulators,
  // masks and the work items of each launch shape
  s->srank = cfg->schedule == LM_SCHEDULE_STABLE_RANK && s->nmat > 0;
  s->mat_param_of.resize(s->nmat);
  for (int id = 0; id < s->nmat; ++id) s->mat_param_of[id] = mat_param[mat_order[id]];
  std::vector<size_t> sr_voff(s->nmat, 0);
  std::vector<std::vector<SrItem>> sr_items;
  size_t off_srv0 = 0, off_srwa = 0, off_srwb = 0, off_sracc = 0, off_srmat = 0, off_active = 0, off_skip = 0,
         off_srank = 0;
  std::vector<size_t> off_sritems;
  if (s->srank) {
    std::map<std::tuple<int, int, bool>, int> shape_launch;
    for (int id = 0; id < s->nmat; ++id) {
      const lm_tensor& p = params[s->mat_param_of[id]];
      int threads = 0;
      const int slots = srank_slots(p.cols, &threads);
      if (slots == 0) {
        delete s;
        return fail(LM_ERR_UNSUPPORTED, "stable-rank schedule: matrix with %lld columns (at most 16384)",
                    (long long)p.cols);
      }
      sr_voff[id] = s->sr_w_elems;
      s->sr_w_elems = align_up(s->sr_w_elems + (size_t)p.cols, 64);
      // rows of 16-byte multiples share a launch per ring-kernel shape, the
      // others per register-kernel shape
      const bool vec4 = p.cols % 4 == 0;
      const auto key = std::make_tuple(vec4 ? srank_ring_shape(p.cols) : slots, threads, vec4);
      auto it = shape_launch.find(key);
      if (it == shape_launch.end()) {
        it = shape_launch.emplace(key, (int)s->sr_launch.size()).first;
        lm_state::SrLaunch L0;
        L0.slots = slots;
        L0.threads = threads;
        L0.vec4 = p.cols % 4 == 0;
        s->sr_launch.push_back(L0);
        sr_items.emplace_back();
      }
      s->sr_launch[it->second].max_cols = std::max<int64_t>(s->sr_launch[it->second].max_cols, p.cols);
      sr_items[it->second].push_back(SrItem{id, 0, (int32_t)p.rows, 0});   // split below
    }
    // Largest launch first: the launches of a pass run concurrently, and the
    // last to finish (whose end no other launch covers) is then the smallest.
    {
      std::vector<int64_t> elems(s->sr_launch.size(), 0);
      for (size_t k = 0; k < sr_items.size(); ++k)
        for (const SrItem& whole : sr_items[k]) elems[k] += (int64_t)whole.nrows * params[s->mat_param_of[whole.m]].cols;
      std::vector<size_t> order(s->sr_launch.size());
      for (size_t k = 0; k < order.size(); ++k) order[k] = k;
      std::stable_sort(order.begin(), order.end(), [&](size_t a, size_t b) { return elems[a] > elems[b]; });
      std::vector<lm_state::SrLaunch> sl;
      std::vector<std::vector<SrItem>> si;
      for (size_t k : order) {
        sl.push_back(s->sr_launch[k]);
        si.push_back(std::move(sr_items[k]));
      }
      s->sr_launch.swap(sl);
      sr_items.swap(si);
    }
    // Work items: runs of rows, sized per launch so that each launch has
    // about eight per block (blocks: two per SM); longer runs mean fewer
    // atomic additions into the M^T u vectors.
    int sms = 0, dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    for (auto& list : sr_items) {
      int64_t total = 0;
      for (const SrItem& whole : list) total += whole.nrows;
      const int64_t per = std::max<int64_t>(kSrankRows,
                                            std::min<int64_t>(8 * kSrankRows, total / (16 * std::max(sms, 1))));
      const int64_t rows_per_item = per / 16 * 16;
      std::vector<SrItem> split;
      for (const SrItem& whole : list)
        for (int64_t r = 0; r < whole.nrows; r += rows_per_item)
          split.push_back(SrItem{whole.m, (int32_t)r, (int32_t)std::min<int64_t>(rows_per_item, whole.nrows - r), 0});
      list.swap(split);
    }
    off_srv0 = ar.add(s->sr_w_elems * sizeof(float));
    off_srwa = ar.add(s->sr_w_elems * sizeof(float));
    off_srwb = ar.add(s->sr_w_elems * sizeof(float));
    off_sracc = ar.add((size_t)s->nmat * (1 + cfg->srank_iters) * sizeof(double));
    off_srmat = ar.add((size_t)s->nmat * sizeof(SrMat));
    off_active = ar.add((size_t)s->nmat);
    off_skip = ar.add((size_t)n);
    off_srank = ar.add((size_t)s->nmat * sizeof(double));
    for (auto& v : sr_items) off_sritems.push_back(ar.add(v.size() * sizeof(SrItem)));
  }

  size_t off_guard_list = 0;
  std::vector<size_t> guard_offs;
  if (s->debug) {
    off_guard_list = ar.add(ar.guards.size() * sizeof(size_t) + sizeof(size_t));
    guard_offs = ar.guards;   // now including the list's own guard
  }
  if (env_is("LM_FAULT", "oom")) {
    delete s;
    return fail(LM_ERR_OOM, "injected allocation failure (LM_FAULT=oom)");
  }
  cudaError_t e = cudaMalloc(&s->base, ar.total);
  if (e != cudaSuccess) {
    delete s;
    return cuda_fail(e, "cudaMalloc(state)");
  }
  s->bytes = ar.total;
  std::vector<char> img(ar.total, 0);
  if (s->debug) {
    for (size_t g : guard_offs) memset(img.data() + g, kGuardByte, kGuardBytes);
    memcpy(img.data() + off_guard_list, guard_offs.data(), guard_offs.size() * sizeof(size_t));
    s->d_guard_offs = reinterpret_cast<size_t*>(s->base + off_guard_list);
    s->n_guards = (int)guard_offs.size();
  }
  char* base = s->base;
  s->mom = reinterpret_cast<float*>(base + off_mom);
  s->d_grads = reinterpret_cast<const void**>(base + off_grads);
  s->d_flags = reinterpret_cast<unsigned*>(base + off_flags);

  for (int d = 0; d < 2; ++d) {
    for (auto& t : lt_all[d]) { t.m = s->mom + s->mom_off[t.pad]; }
    for (auto& t : lt_vec[d]) { t.m = s->mom + s->mom_off[t.pad]; }
    for (auto& t : lt_ema[d]) { t.m = s->mom + s->mom_off[t.pad]; }
    auto put = [&](size_t off, const void* src, size_t bytes) { if (bytes) memcpy(img.data() + off, src, bytes); };
    put(off_lt_all[d], lt_all[d].data(), lt_all[d].size() * sizeof(LionTensor));
    put(off_lc_all[d], lc_all[d].data(), lc_all[d].size() * sizeof(LionChunk));
    put(off_lt_vec[d], lt_vec[d].data(), lt_vec[d].size() * sizeof(LionTensor));
    put(off_lc_vec[d], lc_vec[d].data(), lc_vec[d].size() * sizeof(LionChunk));
    put(off_lt_ema[d], lt_ema[d].data(), lt_ema[d].size() * sizeof(LionTensor));
    put(off_lc_ema[d], lc_ema[d].data(), lc_ema[d].size() * sizeof(LionChunk));
    s->ema[d] = {reinterpret_cast<LionTensor*>(base + off_lt_ema[d]),
                 reinterpret_cast<LionChunk*>(base + off_lc_ema[d]), (int)lc_ema[d].size()};
    s->lion_all[d] = {reinterpret_cast<LionTensor*>(base + off_lt_all[d]),
                      reinterpret_cast<LionChunk*>(base + off_lc_all[d]), (int)lc_all[d].size()};
    s->lion_vec[d] = {reinterpret_cast<LionTensor*>(base + off_lt_vec[d]),
                      reinterpret_cast<LionChunk*>(base + off_lc_vec[d]), (int)lc_vec[d].size()};
    s->lion_grid[d] = lion_grid_size((lm_dtype)d);
  }
  s->vmom = reinterpret_cast<float*>(base + off_v);
  for (int d = 0; d < 2; ++d) {
    for (auto& t : at[d]) {
      t.m = s->mom + s->mom_off[t.pad];
      t.v = s->vmom + s->v_off[t.pad];
    }
    if (!at[d].empty()) memcpy(img.data() + off_at[d], at[d].data(), at[d].size() * sizeof(AdamTensor));
    if (!ac[d].empty()) memcpy(img.data() + off_ac[d], ac[d].data(), ac[d].size() * sizeof(LionChunk));
    s->adam[d] = {reinterpret_cast<AdamTensor*>(base + off_at[d]), reinterpret_cast<LionChunk*>(base + off_ac[d]),
                  (int)ac[d].size()};
  }

  bind_ns(s->ns, base, L, img);
  const bool f32x = s->ns.pieces == 3;   // X_0 and X_K in the fp32 buffer Xf
  const size_t es = f32x ? sizeof(float) : dtype_size(s->ns.xdt);
  for (size_t gi = 0; gi < s->ns.groups.size(); ++gi) {
    const NsGroup& g = s->ns.groups[gi];
    for (int k = 0; k < g.count; ++k) {
      const int id = g.first_mat + k;
      const int pi = mat_param[mat_order[id]];
      const lm_tensor& p = params[pi];
      MatDesc& d = mats[id];
      const size_t xoff = (size_t)k * g.s_pad * g.l_pad * es;
      d.w = p.data;
      d.m = s->mom + s->mom_off[pi];
      d.x = static_cast<char*>(f32x ? g.Xf : g.X[0]) + xoff;
      d.x_final = static_cast<char*>(f32x ? g.Xf : g.X[cfg->ns_steps & 1]) + xoff;
      d.out = nullptr;
      d.norm2 = s->ns.d_norm2 + id;
      d.ldx = g.tall ? g.s_pad : g.l_pad;
      d.grad_slot = pi;
      d.wdt = p.dtype;
      d.odt = p.dtype;
      d.shape_scale = (float)(cfg->shape_scale * std::sqrt((double)std::max(p.rows, p.cols)));
    }
  }
  if (s->nmat) memcpy(img.data() + off_mats, mats.data(), mats.size() * sizeof(MatDesc));
  if (s->srank) {
    float* v0 = reinterpret_cast<float*>(base + off_srv0);
    s->sr_wa = reinterpret_cast<float*>(base + off_srwa);
    s->sr_wb = reinterpret_cast<float*>(base + off_srwb);
    s->sr_acc = reinterpret_cast<double*>(base + off_sracc);
    s->d_sr = reinterpret_cast<SrMat*>(base + off_srmat);
    s->d_active = reinterpret_cast<unsigned char*>(base + off_active);
    s->d_skip = reinterpret_cast<unsigned char*>(base + off_skip);
    s->d_srank = reinterpret_cast<double*>(base + off_srank);
    std::vector<SrMat> srm(s->nmat);
    float* hv0 = reinterpret_cast<float*>(img.data() + off_srv0);
    for (int id = 0; id < s->nmat; ++id) {
      const int pi = s->mat_param_of[id];
      const lm_tensor& p = params[pi];
      // start vector: entry j = 2 * (top 53 bits of SplitMix64 output j) / 2^53 - 1
      uint64_t state = cfg->srank_seed;
      for (int64_t j = 0; j < p.cols; ++j) {
        state += 0x9E3779B97F4A7C15ull;
        uint64_t z = state;
        z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
        z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
        z ^= z >> 31;
        hv0[sr_voff[id] + j] = (float)(2.0 * ((double)(z >> 11) * 0x1.0p-53) - 1.0);
      }
      SrMat& d = srm[id];
      d.M = s->mom + s->mom_off[pi];
      d.v0 = v0 + sr_voff[id];
      d.wa = s->sr_wa + sr_voff[id];
      d.wb = s->sr_wb + sr_voff[id];
      d.acc = s->sr_acc + (size_t)id * (1 + cfg->srank_iters);
      d.rows = p.rows;
      d.cols = p.cols;
      d.mat = id;
      d.param = pi;
    }
    memcpy(img.data() + off_srmat, srm.data(), srm.size() * sizeof(SrMat));
    for (size_t k = 0; k < s->sr_launch.size(); ++k) {
      memcpy(img.data() + off_sritems[k], sr_items[k].data(), sr_items[k].size() * sizeof(SrItem));
      s->sr_launch[k].items = reinterpret_cast<SrItem*>(base + off_sritems[k]);
      s->sr_launch[k].nitems = (int)sr_items[k].size();
    }
  }
  {
    std::vector<ElemChunk> sorted;
    for (int dt = 0; dt < 2; ++dt) {
      for (const ElemChunk& c : echunks_all)
        if (mats[c.mat].wdt == dt) sorted.push_back(c);
      s->n_echunks[dt] = (int)sorted.size() - (dt == 1 ? s->n_echunks[0] : 0);
    }
    if (!sorted.empty()) memcpy(img.data() + off_echunks, sorted.data(), sorted.size() * sizeof(ElemChunk));
  }
  s->d_mats = reinterpret_cast<MatDesc*>(base + off_mats);
  // The last APPLY can write the parameters when they are all bf16 with
  // 16-byte-aligned rows (the epilogue's vector accesses) and NS runs on the
  // tensor cores with at least one iteration.
  s->fuse_final = s->ns.xdt == LM_BF16 && s->ns.pieces == 1 && cfg->ns_steps > 0 && s->nmat > 0;
  for (const MatDesc& d : mats)
    if (d.wdt != LM_BF16 || (d.cols & 7) != 0) s->fuse_final = false;
  if (s->fuse_final) {
    CUtensorMap* hm = reinterpret_cast<CUtensorMap*>(img.data() + off_wmaps);
    for (int id = 0; id < s->nmat && s->fuse_final; ++id)
      if (tc_encode_w_maps(mats[id].w, mats[id].rows, mats[id].cols, hm + 2 * id) != cudaSuccess)
        s->fuse_final = false;   // finalize_kernel writes the parameters instead
    s->d_wmaps = reinterpret_cast<CUtensorMap*>(base + off_wmaps);
  }
  s->d_echunks[0] = reinterpret_cast<ElemChunk*>(base + off_echunks);
  s->d_echunks[1] = s->d_echunks[0] + s->n_echunks[0];

  // Upload tables and zeros (momentum M_{-1} = 0, workspace padding = 0).
  e = cudaMemcpyAsync(base, img.data(), ar.total, cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) {
    cudaFree(s->base);
    delete s;
    return cuda_fail(e, "upload of state tables");
  }
  if ((st = encode_maps(s->ns)) != LM_OK) {
    cudaFree(s->base);
    delete s;
    return st;
  }
  if (s->srank && s->sr_launch.size() >= 2 && (e = create_side_streams(s)) != cudaSuccess) {
    destroy_side_streams(s);
    cudaFree(s->base);
    delete s;
    return cuda_fail(e, "stable-rank side streams");
  }
  s->last_stream = stream;
  *out = s;
  return LM_OK;
}

static lm_status upload_grads(lm_state* s, const lm_tensor* grads, cudaStream_t st) {
  // A step captured into a CUDA graph carries its own pointer upload, and a
  // replay rewrites the device table behind the host's copy: from the first
  // captured step on, every step uploads its pointers.  (The legacy stream
  // cannot be captured.)
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (st != nullptr && cudaStreamIsCapturing(st, &cap) == cudaSuccess && cap != cudaStreamCaptureStatusNone)
    s->captured = true;
  bool same = s->grads_valid && !s->captured;
  for (int i = 0; same && i < s->n; ++i) same = s->h_grads[i] == grads[i].data;
  if (same) return LM_OK;
  s->h_grads.resize(s->n);
  for (int i0 = 0; i0 < s->n; i0 += kPtrsPerUpload) {
    PtrUpload up;
    const int cnt = std::min(kPtrsPerUpload, s->n - i0);
    for (int k = 0; k < cnt; ++k) up.p[k] = grads[i0 + k].data;
    cudaError_t e = timed(&s->prof, LM_KERNEL_OTHER, st,
                          [&]() { return launch_upload_ptrs(s->d_grads + i0, up, cnt, st); });
    if (e != cudaSuccess) {
      s->grads_valid = false;
      return cuda_fail(e, "gradient pointer upload");
    }
  }
  for (int i = 0; i < s->n; ++i) s->h_grads[i] = grads[i].data;
  s->grads_valid = true;
  return LM_OK;
}

}  // extern "C"

// Stable-rank selection on M_{t-1} (Appendix G): srank_iters power-iteration
// passes, then the per-matrix decision into d_active / d_skip.
static lm_status run_srank(lm_state* s, cudaStream_t stream) {
  const int passes = s->cfg.srank_iters;
  Profiler* P = &s->prof;
  cudaError_t e = timed(P, LM_KERNEL_SRANK, stream, [&]() {
    cudaError_t r = cudaMemsetAsync(s->sr_acc, 0, (size_t)s->nmat * (1 + passes) * sizeof(double), stream);
    if (r == cudaSuccess && passes > 1) r = cudaMemsetAsync(s->sr_wa, 0, s->sr_w_elems * sizeof(float), stream);
    return r;
  });
  if (e != cudaSuccess) return cuda_fail(e, "selection buffer reset");
  for (int k = 0; k < passes; ++k) {
    const bool last = k == passes - 1;
    if (k >= 1 && !last) {   // this pass's output vector starts at zero
      float* out = (k & 1) ? s->sr_wb : s->sr_wa;
      e = cudaMemsetAsync(out, 0, s->sr_w_elems * sizeof(float), stream);
      if (e != cudaSuccess) return cuda_fail(e, "selection buffer reset");
    }
    auto launch = [&](const lm_state::SrLaunch& L, cudaStream_t st) {
      if (L.vec4)
        return launch_srank_ring((int)L.max_cols, s->d_sr, L.items, L.nitems, k, last, s->d_flags,
                                 std::min<uint64_t>(kRingWaitNs, s->ns.wait_ns), st);
      return launch_srank_pass(L.slots, L.threads, L.vec4, s->d_sr, L.items, L.nitems, k, last, s->d_flags, st);
    };
    if (s->sr_nside == 0) {
      for (const auto& L : s->sr_launch) {
        e = timed(P, LM_KERNEL_SRANK, stream, [&]() { return launch(L, stream); });
        if (e != cudaSuccess) return cuda_fail(e, "power-iteration launch");
      }
      continue;
    }
    // The launches of one pass touch disjoint matrices: the first runs on the
    // caller's stream, the others on the side streams, all after this pass's
    // reset and before anything the caller enqueues next.
    e = timed(P, LM_KERNEL_SRANK, stream, [&]() {
      cudaError_t r = cudaEventRecord(s->sr_fork, stream);
      for (int q = 0; r == cudaSuccess && q < s->sr_nside; ++q) r = cudaStreamWaitEvent(s->sr_side[q], s->sr_fork, 0);
      for (size_t g = 0; r == cudaSuccess && g < s->sr_launch.size(); ++g)
        r = launch(s->sr_launch[g], g == 0 ? stream : s->sr_side[(g - 1) % s->sr_nside]);
      for (int q = 0; r == cudaSuccess && q < s->sr_nside; ++q) r = cudaEventRecord(s->sr_join[q], s->sr_side[q]);
      for (int q = 0; r == cudaSuccess && q < s->sr_nside; ++q) r = cudaStreamWaitEvent(stream, s->sr_join[q], 0);
      return r;
    });
    if (e != cudaSuccess) return cuda_fail(e, "power-iteration launch");
  }
  e = timed(P, LM_KERNEL_SRANK, stream, [&]() {
    return launch_srank_decide(s->d_sr, s->nmat, s->cfg.srank_alpha, passes - 1, s->d_active, s->d_skip,
                               s->d_srank, s->d_flags, stream);
  });
  if (e != cudaSuccess) return cuda_fail(e, "selection launch");
  return LM_OK;
}

// LM_DEBUG: block k compares guard band k (kGuardBytes at offs[k]) with the
// fill pattern and raises LM_FLAG_GUARD if any byte changed.
__global__ void guard_check_kernel(const unsigned char* base, const size_t* offs, unsigned* flags) {
  const uint4* g = reinterpret_cast<const uint4*>(base + offs[blockIdx.x]);
  const uint32_t pat = 0x01010101u * kGuardByte;
  for (int k = threadIdx.x; k < (int)(kGuardBytes / 16); k += blockDim.x) {
    const uint4 v = g[k];
    if (v.x != pat || v.y != pat || v.z != pat || v.w != pat) atomicOr(flags, LM_FLAG_GUARD);
  }
}

// AdamW over the 1-D parameters of both dtypes (LM_VECTOR_ADAMW).
static lm_status run_adamw(lm_state* s, int64_t t, cudaStream_t stream) {
  AdamConsts ak = adamw_consts(s->cfg, t);
  ak.flags = s->d_flags;
  for (int d = 0; d < 2; ++d) {
    if (s->adam[d].nchunks == 0) continue;
    cudaError_t e = timed(&s->prof, LM_KERNEL_ADAMW, stream, [&]() {
      return launch_adamw((lm_dtype)d, s->adam[d].tensors, s->adam[d].chunks, s->adam[d].nchunks, s->d_grads, ak,
                          stream);
    });
    if (e != cudaSuccess) return cuda_fail(e, "AdamW kernel launch");
  }
  return LM_OK;
}

extern "C" {

lm_status lm_step(lm_state* s, const lm_tensor* grads, int n, int64_t t, void* cuda_stream) {
  if (s == nullptr || grads == nullptr) return fail(LM_ERR_INVALID_ARG, "state/grads is NULL");
  if (n != s->n) return fail(LM_ERR_INVALID_ARG, "n = %d but the state has %d parameters", n, s->n);
  if (t < 0) return fail(LM_ERR_INVALID_ARG, "t must be >= 0");
  lm_status st;
  for (int i = 0; i < n; ++i) {
    if ((st = check_tensor(&grads[i], "grads", i)) != LM_OK) return st;
    if (grads[i].rows != s->params[i].rows || grads[i].cols != s->params[i].cols)
      return fail(LM_ERR_INVALID_ARG, "grads[%d] shape %lldx%lld != param shape %lldx%lld", i,
                  (long long)grads[i].rows, (long long)grads[i].cols, (long long)s->params[i].rows,
                  (long long)s->params[i].cols);
    if (grads[i].dtype != s->params[i].dtype)
      return fail(LM_ERR_DTYPE, "grads[%d] dtype differs from the parameter's", i);
  }
  // device memory: checked once per new gradient pointer
  s->grads_checked.resize(n, nullptr);
  for (int i = 0; i < n; ++i)
    if (grads[i].data != s->grads_checked[i] && (st = check_device_memory(&grads[i], "grads", i, s->device)) != LM_OK)
      return st;
  for (int i = 0; i < n; ++i) s->grads_checked[i] = grads[i].data;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  if ((st = upload_grads(s, grads, stream)) != LM_OK) return st;
  s->last_stream = stream;
  const lm_config& c = s->cfg;
  // Under the stable-rank schedule every step is mixed: matrices take Muon
  // or Lion as the device-side selection says, nothing returns to the host.
  const bool mixed = s->srank;
  const bool muon = mixed || (c.period != 0 && (t % c.period) == 0);
  LionConsts lk = lion_consts(c);
  lk.flags = s->d_flags;
  cudaError_t e;
  Profiler* P = &s->prof;
  s->last_t = t;
  if (mixed) {
    if ((st = run_srank(s, stream)) != LM_OK) return st;
    lk.skip = s->d_skip;
  }
  if (!muon) {
    for (int d = 0; d < 2; ++d) {
      if (s->lion_all[d].nchunks == 0) continue;
      e = timed(P, LM_KERNEL_LION, stream, [&]() {
        return launch_lion((lm_dtype)d, s->lion_all[d].tensors, s->lion_all[d].chunks,
                           s->lion_all[d].nchunks, s->d_grads, lk, s->lion_grid[d], stream);
      });
      if (e != cudaSuccess) return cuda_fail(e, "Lion kernel launch");
    }
    return s->adamw ? run_adamw(s, t, stream) : LM_OK;
  }
  // Muon step: momentum + norm, Lion on the vectors, NS iterations, finalize.
  MuonConsts mk = muon_consts(c);
  mk.flags = s->d_flags;
  if (mixed) mk.active = s->d_active;
  if (s->nmat > 0) {
    e = timed(P, LM_KERNEL_OTHER, stream, [&]() {
      return cudaMemsetAsync(s->ns.d_norm2, 0, (size_t)s->nmat * sizeof(double), stream);
    });
    if (e != cudaSuccess) return cuda_fail(e, "norm reset");
    for (int dt = 0; dt < 2; ++dt) {
      if (s->n_echunks[dt] == 0) continue;
      e = timed(P, LM_KERNEL_MOMENTUM_NORM, stream, [&]() {
        return launch_momentum_norm(s->ns.pieces == 3 ? LM_F32 : s->ns.xdt, (lm_dtype)dt, s->d_mats,
                                    s->d_echunks[dt], s->n_echunks[dt], s->d_grads, mk, 0, stream);
      });
      if (e != cudaSuccess) return cuda_fail(e, "momentum/norm kernel launch");
    }
  }
  // layer sharding: the matrices other ranks own take the momentum update
  // here and their new values from their owners afterwards
  for (int d = 0; d < 2; ++d) {
    if (s->ema[d].nchunks == 0) continue;
    e = timed(P, LM_KERNEL_MOMENTUM_NORM, stream, [&]() {
      return launch_ema((lm_dtype)d, s->ema[d].tensors, s->ema[d].chunks, s->ema[d].nchunks, s->d_grads, lk,
                        s->lion_grid[d], stream);
    });
    if (e != cudaSuccess) return cuda_fail(e, "momentum kernel launch (matrices of other ranks)");
  }
  if (s->adamw) {
    if ((st = run_adamw(s, t, stream)) != LM_OK) return st;
  }
  for (int d = 0; d < 2 && !s->adamw && !mixed; ++d) {
    if (s->lion_vec[d].nchunks == 0) continue;
    e = timed(P, LM_KERNEL_LION, stream, [&]() {
      return launch_lion((lm_dtype)d, s->lion_vec[d].tensors, s->lion_vec[d].chunks,
                         s->lion_vec[d].nchunks, s->d_grads, lk, s->lion_grid[d], stream);
    });
    if (e != cudaSuccess) return cuda_fail(e, "Lion kernel launch (vectors)");
  }
  // mixed step: the Lion table (with the vectors unless AdamW has them)
  // minus the matrices selected for Muon
  for (int d = 0; d < 2 && mixed; ++d) {
    if (s->lion_all[d].nchunks == 0) continue;
    e = timed(P, LM_KERNEL_LION, stream, [&]() {
      return launch_lion((lm_dtype)d, s->lion_all[d].tensors, s->lion_all[d].chunks,
                         s->lion_all[d].nchunks, s->d_grads, lk, s->lion_grid[d], stream);
    });
    if (e != cudaSuccess) return cuda_fail(e, "Lion kernel launch (mixed step)");
  }
  if (s->nmat > 0) {
    const FuseFinal ff{s->d_mats, mk.eM, mk.lam, s->d_wmaps};
    if ((st = run_ns(s->ns, c.ns_steps, s->ns_co.data(), s->d_flags, stream, P, s->fuse_final ? &ff : nullptr,
                     mixed ? s->d_active : nullptr)) != LM_OK)
      return st;
    for (int dt = 0; dt < 2 && !s->fuse_final; ++dt) {
      if (s->n_echunks[dt] == 0) continue;
      e = timed(P, LM_KERNEL_FINALIZE, stream, [&]() {
        return launch_finalize(s->ns.pieces == 3 ? LM_F32 : s->ns.xdt, (lm_dtype)dt, s->d_mats,
                               s->d_echunks[dt], s->n_echunks[dt], mk, 0, s->d_flags, stream);
      });
      if (e != cudaSuccess) return cuda_fail(e, "finalize kernel launch");
    }
  }
  return LM_OK;
}

lm_status lm_set_lr(lm_state* s, double eta_muon, double eta_lion) {
  if (s == nullptr) return fail(LM_ERR_INVALID_ARG, "state is NULL");
  if (!std::isfinite(eta_muon) || !std::isfinite(eta_lion) || eta_muon < 0 || eta_lion < 0)
    return fail(LM_ERR_INVALID_ARG, "learning rates must be finite and >= 0");
  s->cfg.eta_muon = eta_muon;
  s->cfg.eta_lion = eta_lion;
  return LM_OK;
}

lm_status lm_get_selection(lm_state* s, int n, unsigned char* took_muon, double* srank) {
  if (s == nullptr) return fail(LM_ERR_INVALID_ARG, "state is NULL");
  if (n != s->n) return fail(LM_ERR_INVALID_ARG, "n = %d but the state has %d parameters", n, s->n);
  if (s->last_t < 0) return fail(LM_ERR_INVALID_ARG, "no step taken yet");
  const double nan = std::numeric_limits<double>::quiet_NaN();
  std::vector<unsigned char> act(s->nmat, 0);
  std::vector<double> est(s->nmat, nan);
  if (s->srank) {
    cudaError_t e = cudaStreamSynchronize(s->last_stream);
    if (e == cudaSuccess) e = cudaMemcpy(act.data(), s->d_active, (size_t)s->nmat, cudaMemcpyDeviceToHost);
    if (e == cudaSuccess)
      e = cudaMemcpy(est.data(), s->d_srank, (size_t)s->nmat * sizeof(double), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "selection read-back");
  } else {
    const bool muon = s->cfg.period != 0 && (s->last_t % s->cfg.period) == 0;
    std::fill(act.begin(), act.end(), muon ? 1 : 0);
  }
  const bool muon_step = !s->srank && s->cfg.period != 0 && (s->last_t % s->cfg.period) == 0;
  for (int i = 0; i < n; ++i) {
    // under layer sharding a matrix another rank owns also took the Muon
    // step (there, with this rank's momentum update)
    if (took_muon) took_muon[i] = (muon_step && is_matrix(s->params[i])) ? 1 : 0;
    if (srank) srank[i] = nan;
  }
  for (int id = 0; id < s->nmat; ++id) {
    const int pi = s->mat_param_of[id];
    if (took_muon) took_muon[pi] = act[id];
    if (srank) srank[pi] = est[id];
  }
  return LM_OK;
}

lm_status lm_set_adamw_lr(lm_state* s, double lr) {
  if (s == nullptr) return fail(LM_ERR_INVALID_ARG, "state is NULL");
  if (!std::isfinite(lr) || lr < 0) return fail(LM_ERR_INVALID_ARG, "learning rate must be finite and >= 0");
  s->cfg.adamw_lr = lr;
  return LM_OK;
}

lm_status lm_get_second_moment(const lm_state* s, int i, lm_tensor* view) {
  if (s == nullptr || view == nullptr) return fail(LM_ERR_INVALID_ARG, "state/view is NULL");
  if (i < 0 || i >= s->n) return fail(LM_ERR_INVALID_ARG, "index %d out of range", i);
  if (s->v_off[i] < 0) return fail(LM_ERR_INVALID_ARG, "parameter %d has no AdamW second moment", i);
  view->data = s->vmom + s->v_off[i];
  view->rows = s->params[i].rows;
  view->cols = s->params[i].cols;
  view->dtype = LM_F32;
  return LM_OK;
}

lm_status lm_set_second_moment(lm_state* s, int i, const lm_tensor* src, void* cuda_stream) {
  if (s == nullptr || src == nullptr) return fail(LM_ERR_INVALID_ARG, "state/src is NULL");
  if (i < 0 || i >= s->n) return fail(LM_ERR_INVALID_ARG, "index %d out of range", i);
  if (s->v_off[i] < 0) return fail(LM_ERR_INVALID_ARG, "parameter %d has no AdamW second moment", i);
  lm_status st = check_tensor(src, "src", 0);
  if (st != LM_OK) return st;
  if (src->dtype != LM_F32) return fail(LM_ERR_DTYPE, "second-moment source must be fp32");
  if (src->rows != s->params[i].rows || src->cols != s->params[i].cols)
    return fail(LM_ERR_INVALID_ARG, "second-moment source shape differs from the parameter's");
  if ((st = check_device_memory(src, "src", 0, s->device)) != LM_OK) return st;
  const size_t bytes = (size_t)numel(s->params[i]) * sizeof(float);
  if (bytes == 0) return LM_OK;
  cudaError_t e = cudaMemcpyAsync(s->vmom + s->v_off[i], src->data, bytes, cudaMemcpyDeviceToDevice,
                                  static_cast<cudaStream_t>(cuda_stream));
  if (e != cudaSuccess) return cuda_fail(e, "second-moment copy");
  return LM_OK;
}

lm_status lm_get_momentum(const lm_state* s, int i, lm_tensor* view) {
  if (s == nullptr || view == nullptr) return fail(LM_ERR_INVALID_ARG, "state/view is NULL");
  if (i < 0 || i >= s->n) return fail(LM_ERR_INVALID_ARG, "index %d out of range", i);
  view->data = s->mom + s->mom_off[i];
  view->rows = s->params[i].rows;
  view->cols = s->params[i].cols;
  view->dtype = LM_F32;
  return LM_OK;
}

lm_status lm_set_momentum(lm_state* s, int i, const lm_tensor* src, void* cuda_stream) {
  if (s == nullptr || src == nullptr) return fail(LM_ERR_INVALID_ARG, "state/src is NULL");
  if (i < 0 || i >= s->n) return fail(LM_ERR_INVALID_ARG, "index %d out of range", i);
  lm_status st = check_tensor(src, "src", 0);
  if (st != LM_OK) return st;
  if (src->dtype != LM_F32) return fail(LM_ERR_DTYPE, "momentum source must be fp32");
  if (src->rows != s->params[i].rows || src->cols != s->params[i].cols)
    return fail(LM_ERR_INVALID_ARG, "momentum source shape differs from the parameter's");
  if ((st = check_device_memory(src, "src", 0, s->device)) != LM_OK) return st;
  const size_t bytes = (size_t)numel(s->params[i]) * sizeof(float);
  if (bytes == 0) return LM_OK;
  cudaError_t e = cudaMemcpyAsync(s->mom + s->mom_off[i], src->data, bytes, cudaMemcpyDeviceToDevice,
                                  static_cast<cudaStream_t>(cuda_stream));
  if (e != cudaSuccess) return cuda_fail(e, "momentum copy");
  return LM_OK;
}

lm_status lm_get_status(lm_state* s, uint32_t* device_flags) {
  if (s == nullptr || device_flags == nullptr) return fail(LM_ERR_INVALID_ARG, "state/flags is NULL");
  if (s->debug && s->n_guards > 0) {
    count_launch();
    guard_check_kernel<<<s->n_guards, 64, 0, s->last_stream>>>(reinterpret_cast<const unsigned char*>(s->base),
                                                                s->d_guard_offs, s->d_flags);
    cudaError_t g = cudaGetLastError();
    if (g != cudaSuccess) return cuda_fail(g, "guard check launch");
  }
  cudaError_t e = cudaStreamSynchronize(s->last_stream);
  if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
  unsigned f = 0;
  e = cudaMemcpy(&f, s->d_flags, sizeof(unsigned), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "status read");
  e = cudaMemset(s->d_flags, 0, sizeof(unsigned));
  if (e != cudaSuccess) return cuda_fail(e, "status clear");
  *device_flags = f;
  return LM_OK;
}

lm_status lm_profile_enable(lm_state* s, int on) {
  if (s == nullptr) return fail(LM_ERR_INVALID_ARG, "state is NULL");
  s->prof.on = on != 0;
  return LM_OK;
}

lm_status lm_profile_read(lm_state* s, lm_profile* out, int reset) {
  if (s == nullptr || out == nullptr) return fail(LM_ERR_INVALID_ARG, "state/out is NULL");
  Profiler& P = s->prof;
  cudaError_t e = cudaStreamSynchronize(s->last_stream);
  if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
  for (const Profiler::Rec& r : P.recs) {
    float ms = 0.f;
    e = cudaEventElapsedTime(&ms, r.a, r.b);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventElapsedTime");
    P.ms[r.fam] += ms;
    P.n[r.fam] += 1;
  }
  P.recs.clear();
  P.used = 0;
  for (int f = 0; f < LM_KERNEL_FAMILIES; ++f) {
    out->ms[f] = P.ms[f];
    out->launches[f] = P.n[f];
    if (reset) {
      P.ms[f] = 0;
      P.n[f] = 0;
    }
  }
  return LM_OK;
}

lm_status lm_probe_bounded_wait(uint64_t limit_ns, uint32_t* device_flags, void* cuda_stream) {
  if (device_flags == nullptr) return fail(LM_ERR_INVALID_ARG, "device_flags is NULL");
  if (limit_ns == 0 || limit_ns > 10000000000ull) return fail(LM_ERR_INVALID_ARG, "limit_ns must be in (0, 1e10]");
  lm_status st;
  int dev = 0;
  if ((st = check_device(&dev)) != LM_OK) return st;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  unsigned* d = nullptr;
  cudaError_t e = cudaMallocAsync(reinterpret_cast<void**>(&d), sizeof(unsigned), stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaMallocAsync(probe flag)");
  unsigned h = 0;
  e = cudaMemsetAsync(d, 0, sizeof(unsigned), stream);
  if (e == cudaSuccess) e = launch_bounded_wait_probe(limit_ns, d, stream);
  if (e == cudaSuccess) e = cudaMemcpyAsync(&h, d, sizeof(unsigned), cudaMemcpyDeviceToHost, stream);
  cudaFreeAsync(d, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "bounded-wait probe");
  *device_flags = h;
  return (h & LM_FLAG_TIMEOUT) ? fail(LM_ERR_TIMEOUT, "bounded wait gave up after %llu ns",
                                      (unsigned long long)limit_ns)
                               : LM_OK;
}

size_t lm_state_bytes(const lm_state* s) { return s ? (s->mom_elems + s->v_elems) * sizeof(float) : 0; }

size_t lm_workspace_bytes(const lm_state* s) {
  return s ? s->bytes - (s->mom_elems + s->v_elems) * sizeof(float) : 0;
}

void lm_destroy(lm_state* s) {
  if (s == nullptr) return;
  cudaStreamSynchronize(s->last_stream);
  destroy_side_streams(s);
  cudaFree(s->base);
  delete s;
}

}  // extern "C"

// The msign entry points: norm kernel, NS iterations with per-iteration
// coefficients co[0 .. steps-1], output kernel; arguments already checked
// except the tensors and the size limits.
static lm_status msign_impl(const lm_tensor* in, lm_tensor* out, int steps, const std::vector<NsCoeffs>& co,
                            double eps, int precision, void* cuda_stream) {
  lm_status st;
  if ((st = check_tensor(in, "in", 0)) != LM_OK) return st;
  if ((st = check_tensor(out, "out", 0)) != LM_OK) return st;
  if (in->rows < 2 || in->cols < 2) return fail(LM_ERR_INVALID_ARG, "msign needs rows, cols >= 2");
  if (out->rows != in->rows || out->cols != in->cols) return fail(LM_ERR_INVALID_ARG, "out shape differs from in");
  if (std::max(in->rows, in->cols) > 1000000 || std::min(in->rows, in->cols) > 65536)
    return fail(LM_ERR_UNSUPPORTED, "matrix too large for lm_msign_ns");
  int dev = 0;
  if ((st = check_device(&dev)) != LM_OK) return st;
  if ((st = check_device_memory(in, "in", 0, dev)) != LM_OK) return st;
  if ((st = check_device_memory(out, "out", 0, dev)) != LM_OK) return st;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);

  NsEngine E;
  E.xdt = precision == LM_F32 ? LM_F32 : LM_BF16;
  E.pieces = precision == LM_NS_F32_TC ? 3 : 1;
  const lm_dtype xio = E.pieces == 3 ? LM_F32 : E.xdt;   // X_0 / X_K buffer dtype
  std::vector<std::vector<int>> members;
  plan_groups({{in->rows, in->cols}}, E.xdt, E.groups, members);
  Arena ar;
  NsLayout L;
  layout_ns(E.groups, E.xdt, 1, ar, L, E.batches, E.pieces, env_tiles_mode());
  E.pdl = !env_is("LM_PDL", "0");
  E.fold = !env_is("LM_NS_FOLD", "0");
  E.wait_ns = env_wait_limit_ns();
  const size_t off_mat = ar.add(sizeof(MatDesc));
  MatDesc d;
  memset(&d, 0, sizeof(d));
  d.rows = in->rows;
  d.cols = in->cols;
  std::vector<ElemChunk> et;
  build_elem_chunks({d}, et);
  const size_t off_et = ar.add(et.size() * sizeof(ElemChunk));
  const size_t off_flags = ar.add(sizeof(unsigned));

  char* base = nullptr;
  cudaError_t e = cudaMallocAsync(reinterpret_cast<void**>(&base), ar.total, stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaMallocAsync(msign workspace)");
  std::vector<char> img(ar.total, 0);
  bind_ns(E, base, L, img);
  const NsGroup& g = E.groups[0];
  d.w = in->data;
  d.m = nullptr;
  d.x = E.pieces == 3 ? g.Xf : g.X[0];
  d.x_final = E.pieces == 3 ? g.Xf : g.X[steps & 1];
  d.out = out->data;
  d.norm2 = E.d_norm2;
  d.ldx = g.tall ? g.s_pad : g.l_pad;
  d.grad_slot = 0;
  d.wdt = in->dtype;
  d.odt = out->dtype;
  d.shape_scale = 1.f;
  memcpy(img.data() + off_mat, &d, sizeof(d));
  memcpy(img.data() + off_et, et.data(), et.size() * sizeof(ElemChunk));
  auto cleanup = [&](lm_status r) {
    cudaFreeAsync(base, stream);
    return r;
  };
  e = cudaMemcpyAsync(base, img.data(), ar.total, cudaMemcpyHostToDevice, stream);
  if (e != cudaSuccess) return cleanup(cuda_fail(e, "msign table upload"));
  if ((st = encode_maps(E)) != LM_OK) return cleanup(st);
  MuonConsts mk;
  memset(&mk, 0, sizeof(mk));
  mk.eps = (float)eps;
  mk.ns_steps = steps;
  MatDesc* dm = reinterpret_cast<MatDesc*>(base + off_mat);
  ElemChunk* de = reinterpret_cast<ElemChunk*>(base + off_et);
  unsigned* dflags = reinterpret_cast<unsigned*>(base + off_flags);
  mk.flags = dflags;
  e = launch_momentum_norm(xio, in->dtype, dm, de, (int)et.size(), nullptr, mk, 1, stream);
  if (e != cudaSuccess) return cleanup(cuda_fail(e, "norm kernel launch"));
  if ((st = run_ns(E, steps, co.data(), dflags, stream)) != LM_OK) return cleanup(st);
  e = launch_finalize(xio, out->dtype, dm, de, (int)et.size(), mk, 1, dflags, stream);
  if (e != cudaSuccess) return cleanup(cuda_fail(e, "output kernel launch"));
  // the call's status word: read back before the workspace goes
  unsigned hflags = 0;
  e = cudaMemcpyAsync(&hflags, dflags, sizeof(unsigned), cudaMemcpyDeviceToHost, stream);
  cudaFreeAsync(base, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "msign status read");
  if (hflags & LM_FLAG_TIMEOUT)
    return fail(LM_ERR_TIMEOUT, "a bounded device wait gave up; out was not written (LM_FLAG_TIMEOUT)");
  return LM_OK;
}

extern "C" {

lm_status lm_msign_ns(const lm_tensor* in, lm_tensor* out, int steps, double a, double b, double c,
                      double eps, int precision, void* cuda_stream) {
  if (in == nullptr || out == nullptr) return fail(LM_ERR_INVALID_ARG, "in/out is NULL");
  if (steps < 0 || steps > 64) return fail(LM_ERR_INVALID_ARG, "steps must be in [0, 64]");
  if (!std::isfinite(a) || !std::isfinite(b) || !std::isfinite(c) || !std::isfinite(eps) || eps < 0)
    return fail(LM_ERR_INVALID_ARG, "coefficients must be finite, eps >= 0");
  if (precision != LM_BF16 && precision != LM_F32 && precision != LM_NS_F32_TC)
    return fail(LM_ERR_INVALID_ARG, "precision must be LM_BF16, LM_F32 or LM_NS_F32_TC");
  return msign_impl(in, out, steps, ns_schedule(steps, nullptr, a, b, c, eps), eps, precision, cuda_stream);
}

lm_status lm_msign_ns_coeffs(const lm_tensor* in, lm_tensor* out, int steps, const double* coeffs, double eps,
                             int precision, void* cuda_stream) {
  if (in == nullptr || out == nullptr) return fail(LM_ERR_INVALID_ARG, "in/out is NULL");
  if (steps < 0 || steps > 64) return fail(LM_ERR_INVALID_ARG, "steps must be in [0, 64]");
  if (steps > 0 && coeffs == nullptr) return fail(LM_ERR_INVALID_ARG, "coeffs is NULL");
  for (int k = 0; k < 3 * steps; ++k)
    if (!std::isfinite(coeffs[k])) return fail(LM_ERR_INVALID_ARG, "coeffs[%d] is not finite", k);
  if (!std::isfinite(eps) || eps < 0) return fail(LM_ERR_INVALID_ARG, "eps must be finite and >= 0");
  if (precision != LM_BF16 && precision != LM_F32 && precision != LM_NS_F32_TC)
    return fail(LM_ERR_INVALID_ARG, "precision must be LM_BF16, LM_F32 or LM_NS_F32_TC");
  return msign_impl(in, out, steps, ns_schedule(steps, coeffs, 0, 0, 0, eps), eps, precision, cuda_stream);
}

}  // extern "C"
