// Wide-tile tensor-core Newton-Schulz phases for sm_103a (bf16 operands,
// fp32 accumulators in TMEM, CTA pairs with cta_group::2).
//
// A tile is one or two 256-column halves of a 256-row output block.  For a
// two-half tile the pair stages, per 64-deep K block, one A box of its rows
// and two B boxes (one per half), and issues two N = 256 MMAs that read the
// same A box: 48 KB per CTA for 8.4 MFLOP, against 32 KB for 4.2 MFLOP with
// one half.  Staged bytes per FLOP, which is what holds the narrow kernel
// (lm_ns_tc.cu) below the tensor pipe's rate, drop by a quarter (by half on a
// tile whose first half is diagonal, where B0 is the A box itself).
//
// The phases are those of Section 2's iteration, as in lm_ns_tc.cu: GRAM
// A = X X^T (tall: X^T X), POLY B = b A + c A A, APPLY X' = a X + B X
// (tall: a X + X B), with only the upper 256 x 256 blocks of A and B stored.
// A symmetric tile pairs block (tm, tn) with (tm, tn + 1), so every stored
// block is computed once; an APPLY tile pairs column blocks 2k and 2k + 1.
//
// TMEM holds two 256-column accumulator halves used as a ring: a one-half
// tile takes the next half (so the epilogue of one tile overlaps the main
// loop of the next), a two-half tile takes both.  Per K block the layouts of
// A, B0 and B1 (K-major rows or MN-major columns of a stored matrix) are fixed
// over ranges of K (TilePlanW), and the producer and MMA loops are compiled
// per layout combination.
//
// CTA roles (352 threads, one CTA per SM):
//   warp 0    TMA producer (one lane), 3-stage ring of 48 KB; both CTAs'
//             copies signal CTA 0's full barrier
//   warp 1    TMEM allocator (both CTAs) + MMA issuer (CTA 0, one lane)
//   warps 2-9 epilogue: warp (q, hw) serves TMEM lane quadrant q and columns
//             [128 hw, 128 hw + 128) of each half, as two 64-column boxes
//   warp 10   aux loader: TMA of the A (POLY) or X (APPLY) boxes the
//             epilogue combines with the accumulator, into four 16 KB slots
// The slots double as the store staging: an epilogue warp writes its 32 rows
// of a box over the aux values and stores them by TMA.  The last APPLY of a
// Muon step can instead update the parameters W <- W - eta_M (s X_K +
// lambda W) (Algorithm 1, Muon branch) from the box.  Every wait is bounded.
#include <cuda_bf16.h>

#include "lm_ns_tc_shared.cuh"

namespace lm {
namespace {

using namespace tc;
using namespace tcs;

constexpr int kWStageBytes = kABytes + 2 * kBBytes;   // A | B0 | B1
constexpr int kTmemColsW = 2 * BN;
// Shared memory per phase: POLY / APPLY: a 3-stage ring and four 16 KB
// slots for the aux boxes; GRAM (no aux boxes): a 4-stage ring and two
// slots of store staging.
template <bool kGram>
struct WLayout {
  static constexpr int kStages = kGram ? 4 : 3;
  static constexpr int kSlots = kGram ? 2 : 4;
  static constexpr size_t kSlotOffset = (size_t)kStages * kWStageBytes;
  static constexpr size_t kBarOffset = kSlotOffset + (size_t)kSlots * kAuxBoxBytes;
  static constexpr size_t kSmemBytes = 1024 /*align slack*/ + kBarOffset + 512;
};
constexpr int kMaxWStages = 4;

__device__ __forceinline__ int tile_halves(const NsTile& t) { return t.nh == 2 ? 2 : 1; }

// Operand layouts over a range of K blocks: A, and B of each half, K-major
// (rows of a stored matrix) or MN-major (its columns).
struct OpSegW {
  int kb_end;
  bool a_mn, b0_mn, b1_mn;
  const CUtensorMap* ma;
  const CUtensorMap* mb0;
  const CUtensorMap* mb1;
};
struct TilePlanW {
  int nseg;
  int kb_start;
  OpSegW seg[4];
};
__device__ __forceinline__ void planw_push(TilePlanW& P, int kb_end, bool a, bool b0, bool b1, const CUtensorMap* ma,
                                           const CUtensorMap* mb0, const CUtensorMap* mb1) {
  const int prev = P.nseg ? P.seg[P.nseg - 1].kb_end : P.kb_start;
  if (kb_end <= prev) return;
  P.seg[P.nseg++] = OpSegW{kb_end, a, b0, b1, ma, mb0, mb1};
}
// Row block tm of a stored symmetric matrix reads K blocks at or after
// 4 tm K-major from its stored tiles and those before as transposed stored
// tiles (MN-major); B half h covers column block tn + h.
__device__ __forceinline__ TilePlanW tile_plan_w(int phase, const NsGroup& g, const TcGroupMaps& mp, int cur,
                                                 const NsTile& t) {
  TilePlanW P;
  P.nseg = 0;
  P.kb_start = 0;
  if (phase == NS_GRAM) {
    const int nk = g.l_pad / BK;
    const int kb_end = t.kb1 != 0 ? (int)t.kb1 : nk;
    P.kb_start = t.kb1 != 0 ? (int)t.kb0 : 0;
    if (g.tall) planw_push(P, kb_end, true, true, true, &mp.xmn[cur], &mp.xmn[cur], &mp.xmn[cur]);
    else planw_push(P, kb_end, false, false, false, &mp.xk[cur], &mp.xk[cur], &mp.xk[cur]);
    return P;
  }
  const int nk = g.s_pad / BK;
  const int ka = min(t.tm * (BM / BK), nk);
  const int kn0 = min(t.tn * (BN / BK), nk);
  const int kn1 = min((t.tn + 1) * (BN / BK), nk);
  if (phase == NS_POLY) {   // A-operand rows tm, B rows tn and tn + 1 (tn >= tm)
    planw_push(P, ka, true, true, true, &mp.amn, &mp.amn, &mp.amn);
    planw_push(P, kn0, false, true, true, &mp.a, &mp.amn, &mp.amn);
    planw_push(P, kn1, false, false, true, &mp.a, &mp.a, &mp.amn);
    planw_push(P, nk, false, false, false, &mp.a, &mp.a, &mp.a);
  } else if (!g.tall) {     // rows tm of B, X MN-major
    planw_push(P, ka, true, true, true, &mp.bmn, &mp.xmn[cur], &mp.xmn[cur]);
    planw_push(P, nk, false, true, true, &mp.b, &mp.xmn[cur], &mp.xmn[cur]);
  } else {                  // rows of X K-major, rows tn and tn + 1 of B
    planw_push(P, kn0, false, true, true, &mp.xk[cur], &mp.bmn, &mp.bmn);
    planw_push(P, kn1, false, false, true, &mp.xk[cur], &mp.b, &mp.bmn);
    planw_push(P, nk, false, false, false, &mp.xk[cur], &mp.b, &mp.b);
  }
  return P;
}

template <int kStages>
struct RingW {
  int stage;
  uint32_t ph;
  int armed[kStages];   // CTA 0: parity of the last phase armed per stage, -1 none
};

// One operand box: a 64 (K) x 128 K-major box, or one 4-D box filling both
// 64-wide MN-major swizzle atoms of a 128-wide half.
template <bool MN>
__device__ __forceinline__ void load_box(void* dst, const CUtensorMap* map, uint32_t bar, int k0, int row, int mat) {
  if (!MN) tma_load_3d(dst, map, bar, k0, row, mat);
  else tma_load_4d(dst, map, bar, 0, k0, row >> 6, mat);
}

// Producer loop over K blocks [kb0, kb1) of one tile with fixed layouts.
// same0 / same1: B half 0 / 1 is the A box itself (a diagonal block).
template <bool AMN, bool B0MN, bool B1MN, int kWStages>
__device__ __forceinline__ bool produce_w(RingW<kWStages>& R, ProducerLog<kWStages>& log, uint8_t* smem, uint64_t* full,
                                          uint64_t* empty, volatile int* abort_flag, uint64_t wait_ns, uint32_t rank,
                                          int kb0, int kb1, const OpSegW& S, int row_a, int col_b0, int mat, int nh,
                                          bool same0, bool same1) {
  const uint32_t own = (uint32_t)kABytes + (same0 ? 0u : (uint32_t)kBBytes) +
                       ((nh == 2 && !same1) ? (uint32_t)kBBytes : 0u);
  for (int kb = kb0; kb < kb1; ++kb) {
    if (!mbar_wait(&empty[R.stage], R.ph ^ 1u, abort_flag, wait_ns)) return false;
    uint8_t* sa = smem + (size_t)R.stage * kWStageBytes;
    const uint32_t fb = peer_addr(&full[R.stage], 0);
    if (rank == 0) {
      mbar_arrive_expect_tx(&full[R.stage], 2u * own);
      R.armed[R.stage] = (int)R.ph;
    }
    log.bytes[R.stage] = own;
    log.n += 1u;
    const int k0 = kb * BK;
    load_box<AMN>(sa, S.ma, fb, k0, row_a, mat);
    if (!same0) load_box<B0MN>(sa + kABytes, S.mb0, fb, k0, col_b0, mat);
    if (nh == 2 && !same1) load_box<B1MN>(sa + kABytes + kBBytes, S.mb1, fb, k0, col_b0 + BN, mat);
    if (++R.stage == kWStages) {
      R.stage = 0;
      R.ph ^= 1u;
    }
  }
  return true;
}

// MMA issue over K blocks [kb0, kb1): per 16-deep step one N = 256 MMA per
// half into accumulators d0 / d1, both reading the same A descriptor.
template <bool AMN, bool B0MN, bool B1MN, int kWStages>
__device__ __forceinline__ bool mma_w(int& stage, uint32_t& ph, uint8_t* smem, uint64_t* full, uint64_t* empty,
                                      volatile int* abort_flag, uint64_t wait_ns, int kb0, int kb1, int kb_first,
                                      uint32_t d0, uint32_t d1, int nh, bool same0, bool same1) {
  constexpr uint32_t idesc0 = make_idesc(BM, BN, AMN, B0MN);
  constexpr uint32_t idesc1 = make_idesc(BM, BN, AMN, B1MN);
  for (int kb = kb0; kb < kb1; ++kb) {
    if (!mbar_wait(&full[stage], ph, abort_flag, wait_ns)) return false;
    tc_fence_after();
    const uint32_t sa = smem_u32(smem + (size_t)stage * kWStageBytes);
    const uint32_t sb0 = same0 ? sa : sa + kABytes;
    const uint32_t sb1 = same1 ? sa : sa + kABytes + kBBytes;
#pragma unroll
    for (int kk = 0; kk < BK / 16; ++kk) {
      const uint64_t adesc = AMN ? sw128_desc(sa + kk * 2048, 64 * BK * 2, 1024) : sw128_desc(sa + kk * 32, 16, 1024);
      const uint64_t b0 = B0MN ? sw128_desc(sb0 + kk * 2048, 64 * BK * 2, 1024) : sw128_desc(sb0 + kk * 32, 16, 1024);
      const uint32_t acc = (kb != kb_first || kk != 0) ? 1u : 0u;
      umma_bf16(d0, adesc, b0, idesc0, acc);
      if (nh == 2) {
        const uint64_t b1 =
            B1MN ? sw128_desc(sb1 + kk * 2048, 64 * BK * 2, 1024) : sw128_desc(sb1 + kk * 32, 16, 1024);
        umma_bf16(d1, adesc, b1, idesc1, acc);
      }
    }
    umma_commit_pair(&empty[stage]);
    if (++stage == kWStages) {
      stage = 0;
      ph ^= 1u;
    }
  }
  return true;
}

// The layout combinations the plans produce: (A, B0, B1) MN-major flags
// 111, 011, 001, 000.
#define LM_W_DISPATCH(FN, S, ...)                                                      \
  ((S).a_mn ? FN<true, true, true, kWStages>(__VA_ARGS__)                              \
            : ((S).b0_mn ? FN<false, true, true, kWStages>(__VA_ARGS__)                \
                         : ((S).b1_mn ? FN<false, false, true, kWStages>(__VA_ARGS__)  \
                                      : FN<false, false, false, kWStages>(__VA_ARGS__))))

__device__ __forceinline__ float bf_lo_w(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf_hi_w(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

// kMasked: per-matrix mask (stable-rank selection); kSplit: the launch's Gram
// tiles include split-K parts (those are one-half tiles).
template <bool kMasked, bool kSplit, bool kGram>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    ns_wide_kernel(const __grid_constant__ TcParams p) {
  using Lw = WLayout<kGram>;
  constexpr int kWStages = Lw::kStages;
  constexpr int kSlots = Lw::kSlots;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* slots = smem + Lw::kSlotOffset;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + Lw::kBarOffset);
  uint64_t* empty = full + kWStages;
  uint64_t* accfull = empty + kWStages;     // per accumulator half
  uint64_t* accempty = accfull + 2;
  uint64_t* aux_full = accempty + 2;        // per slot
  uint64_t* aux_empty = aux_full + kSlots;
  uint64_t* done = aux_empty + kSlots;
  ProducerLog<kWStages>* log = reinterpret_cast<ProducerLog<kWStages>*>(done + 1);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(log + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint32_t* stop_word = reinterpret_cast<uint32_t*>(tmem_slot + 2);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int phase = p.phase;
  const int cur = p.iter & 1;
  const uint32_t rank = cluster_rank();
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  const bool aux_phase = !kGram;
  int w_begin = p.offsets ? p.offsets[pair] : pair;
  const int w_end = p.offsets ? p.offsets[pair + 1] : p.ntiles;
  const int w_step = p.offsets ? 1 : npairs;

  if constexpr (kMasked) {
    // the mask comes from a kernel this launch may overlap: wait for it first
    griddep_wait();
    int any = 0;
    for (int w = w_begin + (int)threadIdx.x * w_step; !any && w < w_end; w += (int)blockDim.x * w_step)
      any = tile_active(p, p.tiles[w]) ? 1 : 0;
    if (!__syncthreads_or(any)) {
      griddep_launch_dependents();
      return;
    }
  }

  if (threadIdx.x == 0) {
    for (int s = 0; s < kWStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int h = 0; h < 2; ++h) {
      mbar_init(&accfull[h], 1);
      mbar_init(&accempty[h], 2 * kEpiWarps);
    }
    for (int s = 0; s < kSlots; ++s) {
      mbar_init(&aux_full[s], 1);
      mbar_init(&aux_empty[s], 4);   // the four quadrant warps sharing the slot
    }
    mbar_init(done, 1);
    log->n = 0;
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemColsW);
    tmem_relinquish();
  }
  if (pair_start(p, stop_word, rank)) w_begin = w_end;   // an earlier launch gave up: no tiles
  const uint32_t tmem_base = *tmem_slot;
  const uint64_t wait_ns = p.wait_ns;

  auto give_up = [&]() {
    *abort_flag = 1;
    atomicOr(p.flags, LM_FLAG_TIMEOUT);
  };

  RingW<kWStages> R;   // producer lane: ring position and armed phases
  R.stage = 0;
  R.ph = 0;
  for (int s = 0; s < kWStages; ++s) R.armed[s] = -1;

  if (warp == 0) {
    // ------------------------------ producer ------------------------------
    if (lane == 0) {
      bool ok = true;
      for (int w = w_begin; ok && w < w_end; w += w_step) {
        const NsTile t = p.tiles[w];
        if (kMasked && !tile_active(p, t)) continue;
        const NsGroup& g = p.groups[t.group];
        const int nh = tile_halves(t);
        const TilePlanW P = tile_plan_w(phase, g, p.maps[t.group], cur, t);
        const int row_a = t.tm * BM + (int)rank * kHalf;
        const int col_b0 = t.tn * BN + (int)rank * kHalf;
        int kb0 = P.kb_start;
        for (int sg = 0; ok && sg < P.nseg; ++sg) {
          const OpSegW& S = P.seg[sg];
          const bool same0 = S.ma == S.mb0 && t.tm == t.tn;
          const bool same1 = S.ma == S.mb1 && t.tm == t.tn + 1;
          ok = LM_W_DISPATCH(produce_w, S, R, *log, smem, full, empty, abort_flag, wait_ns, rank, kb0, S.kb_end, S,
                             row_a, col_b0, t.mat, nh, same0, same1);
          kb0 = S.kb_end;
        }
        if (!ok) give_up();
      }
    }
  } else if (warp == 1) {
    // ------------------------------ MMA issuer -----------------------------
    if (lane == 0 && rank == 0) {
      int stage = 0;
      uint32_t ph = 0;
      uint32_t hc = 0;   // accumulator halves taken so far: half hc & 1, use hc >> 1
      bool ok = true;
      for (int w = w_begin; ok && w < w_end; w += w_step) {
        const NsTile t = p.tiles[w];
        if (kMasked && !tile_active(p, t)) continue;
        const NsGroup& g = p.groups[t.group];
        const int nh = tile_halves(t);
        const TilePlanW P = tile_plan_w(phase, g, p.maps[t.group], cur, t);
        for (int i = 0; ok && i < nh; ++i) {
          const uint32_t c = hc + (uint32_t)i;
          ok = mbar_wait(&accempty[c & 1u], ((c >> 1) & 1u) ^ 1u, abort_flag, wait_ns);
        }
        if (!ok) {
          give_up();
          break;
        }
        tc_fence_after();
        const uint32_t d0 = tmem_base + (hc & 1u) * BN, d1 = tmem_base + ((hc + 1u) & 1u) * BN;
        int kb0 = P.kb_start;
        for (int sg = 0; ok && sg < P.nseg; ++sg) {
          const OpSegW& S = P.seg[sg];
          const bool same0 = S.ma == S.mb0 && t.tm == t.tn;
          const bool same1 = S.ma == S.mb1 && t.tm == t.tn + 1;
          ok = LM_W_DISPATCH(mma_w, S, stage, ph, smem, full, empty, abort_flag, wait_ns, kb0, S.kb_end, P.kb_start,
                             d0, d1, nh, same0, same1);
          kb0 = S.kb_end;
        }
        if (!ok) {
          give_up();
          break;
        }
        for (int i = 0; i < nh; ++i) umma_commit_pair(&accfull[(hc + (uint32_t)i) & 1u]);
        hc += (uint32_t)nh;
      }
      // all issued MMAs complete before TMEM is released or the CTAs leave
      umma_commit_local(done);
      volatile int never = 0;
      mbar_wait(done, 0, &never, kCleanupWaitNs);
    }
  } else if (warp == kAuxWarp) {
    // --------------------------- aux box loader ---------------------------
    if (lane == 0 && aux_phase) {
      uint32_t hu = 0;   // tile halves loaded so far (every slot is used once per half)
      int armed[kSlots];   // parity of each slot's last armed load
      for (int s = 0; s < kSlots; ++s) armed[s] = -1;
      bool ok = true;
      for (int w = w_begin; ok && w < w_end; w += w_step) {
        const NsTile t = p.tiles[w];
        if (kMasked && !tile_active(p, t)) continue;
        const TcGroupMaps& mp = p.maps[t.group];
        const CUtensorMap* map = (phase == NS_POLY) ? &mp.a : &mp.xk[cur];
        const int nh = tile_halves(t);
        const int row0 = t.tm * BM + (int)rank * kHalf;
        for (int i = 0; ok && i < nh; ++i, ++hu) {
          for (int s = 0; ok && s < kSlots; ++s) {
            if (!mbar_wait(&aux_empty[s], (hu & 1u) ^ 1u, abort_flag, wait_ns)) {
              give_up();
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&aux_full[s], kAuxBoxBytes);
            armed[s] = (int)(hu & 1u);
            tma_load_3d_local(slots + s * kAuxBoxBytes, map, &aux_full[s], (t.tn + i) * BN + 64 * s, row0, t.mat);
          }
        }
      }
      if (!ok) {
        // let the loads already issued land before the CTA leaves
        volatile int never = 0;
        for (int s = 0; s < kSlots; ++s)
          if (armed[s] >= 0) mbar_wait(&aux_full[s], (uint32_t)armed[s], &never, kCleanupWaitNs);
      }
    }
  } else {
    // ------------------------------ epilogue -------------------------------
    // Warp (q, hw): rows [32 q, 32 q + 32) of the CTA's 128, columns
    // [128 hw, 128 hw + 128) of each half, as the boxes in slots 2 hw, 2 hw + 1.
    const int q = warp & 3;
    const int hw = (warp - 2) >> 2;
    const int row = q * 32 + lane;   // row of the CTA's 128-row block
    uint32_t hc = 0, hu = 0;
    bool stop = false;
    for (int w = w_begin; !stop && w < w_end; w += w_step) {
      const NsTile t = p.tiles[w];
      if (kMasked && !tile_active(p, t)) continue;
      const NsGroup& g = p.groups[t.group];
      const int nh = tile_halves(t);
      const bool fused = phase == NS_APPLY && p.fuse.mats != nullptr;
      const MatDesc* fd = fused ? &p.fuse.mats[g.first_mat + t.mat] : nullptr;
      // a tile whose epilogue starts after a give-up was recorded leaves W alone
      const unsigned flags_now = fused && lane == 0 ? *reinterpret_cast<volatile unsigned*>(p.flags) : 0u;
      const bool write_w = fused && __shfl_sync(0xffffffffu, flags_now, 0) == 0u;
      float nscale = 1.f;
      if (p.iter == 0) {
        const float n = (float)sqrt(p.norm2[g.first_mat + t.mat]) + p.co.eps;
        nscale = (phase == NS_GRAM) ? 1.f / (n * n) : (phase == NS_APPLY ? 1.f / n : 1.f);
      }
      // output extents: s x s (GRAM, POLY), s x l (APPLY wide), l x s (APPLY tall)
      const bool apply_tall = phase == NS_APPLY && g.tall;
      const int nrows = apply_tall ? g.l : g.s;
      const int row_lim = apply_tall ? g.l_pad : g.s_pad;
      const int ncols = (phase == NS_APPLY) ? (g.tall ? g.s : g.l) : g.s;
      const int jmax = (phase == NS_APPLY) ? (g.tall ? g.s_pad : g.l_pad) : g.s_pad;
      const int r0 = t.tm * BM + (int)rank * kHalf + q * 32;   // first row of this warp
      const int i_row = r0 + lane;
      const bool warp_in = r0 < row_lim;
      const bool split = kSplit && phase == NS_GRAM && t.slot != 0;
      if (fused && lane == 0 && q == 0 && hw == 0 && rank == 0 && t.tm == 0 && t.tn == 0 &&
          !isfinite((float)sqrt(p.norm2[g.first_mat + t.mat])))
        atomicOr(p.flags, LM_FLAG_NONFINITE);
      for (int i = 0; i < nh; ++i, ++hc, ++hu) {
        const uint32_t half = hc & 1u;
        bool ok = true;
        if (lane == 0) ok = mbar_wait(&accfull[half], (hc >> 1) & 1u, abort_flag, wait_ns);
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        if (!ok) {
          if (lane == 0) give_up();
          stop = true;
          break;
        }
        tc_fence_after();
        const int jh = (t.tn + i) * BN;   // first output column of this half
        for (int bb = 0; bb < 2; ++bb) {
          const int s = 2 * hw + bb;
          const int jb = jh + 64 * s;     // first output column of the box
          // aux phases: the box's own slot; GRAM: slot hw, its two boxes in turn
          uint8_t* box = slots + (kSlots == 4 ? s : hw) * kAuxBoxBytes;
          if (aux_phase) {
            if (lane == 0) ok = mbar_wait(&aux_full[s], hu & 1u, abort_flag, wait_ns);
            ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
            if (!ok) {
              if (lane == 0) give_up();
              stop = true;
              break;
            }
          } else if (!split) {
            // this warp's rows of the slot: its previous store has read them
            if (lane == 0) {
              if (kSlots == 4) asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
              else asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
            }
            __syncwarp();
          }
          for (int c = 0; c < 2; ++c) {
            uint32_t r[32];
            __syncwarp();   // tcgen05.ld is warp-collective: reconverge first
            tmem_ld32(tmem_base + ((uint32_t)(q * 32) << 16) + half * BN + (uint32_t)(64 * s + 32 * c), r);
            const int j0 = jb + 32 * c;
            if (!warp_in || j0 >= jmax) continue;
            if (split) {
              // partial Gram product of a split tile: its own fp32 workspace tile
              float* wrow = p.split_ws + (size_t)(t.slot - 1) * (BM * BN) + (size_t)((int)rank * kHalf + row) * BN +
                            64 * s + 32 * c;
#pragma unroll
              for (int e = 0; e < 32; e += 4) {
                float o[4];
#pragma unroll
                for (int u = 0; u < 4; ++u)
                  o[u] = (i_row < nrows && j0 + e + u < ncols) ? __uint_as_float(r[e + u]) * nscale : 0.f;
                *reinterpret_cast<float4*>(wrow + e) = make_float4(o[0], o[1], o[2], o[3]);
              }
              continue;
            }
            // 16-byte chunk k of a box row sits at chunk position k ^ (row mod 8)
            uint4* brow = reinterpret_cast<uint4*>(box + row * 128);
            float v[32];
            if (aux_phase) {
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                const uint4 a4 = brow[(4 * c + u) ^ (row & 7)];
                const uint32_t aw[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  v[u * 8 + 2 * e] = bf_lo_w(aw[e]);
                  v[u * 8 + 2 * e + 1] = bf_hi_w(aw[e]);
                }
              }
            }
#pragma unroll
            for (int e = 0; e < 32; ++e) {
              const float acc = __uint_as_float(r[e]);
              float o;
              if (phase == NS_GRAM) o = acc * nscale;
              else if (phase == NS_POLY) o = p.co.b * v[e] + p.co.c * acc;
              else o = __fmaf_rn(p.co.a, v[e], acc) * nscale;   // the same rounding as ns_tc_kernel
              v[e] = (i_row < nrows && j0 + e < ncols) ? o : 0.f;
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
              brow[(4 * c + u) ^ (row & 7)] =
                  make_uint4(pack_bf2(v[u * 8 + 0], v[u * 8 + 1]), pack_bf2(v[u * 8 + 2], v[u * 8 + 3]),
                             pack_bf2(v[u * 8 + 4], v[u * 8 + 5]), pack_bf2(v[u * 8 + 6], v[u * 8 + 7]));
          }
          if (bb == 1) {
            // every TMEM column of this half this warp reads has been read
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(peer_addr(&accempty[half], 0));
          }
          fence_proxy_async_smem();
          __syncwarp();
          const bool box_in = warp_in && jb < jmax && !split;
          if (fused) {
            // W <- W - eta_M (s X_K + lambda W) from this warp's 32 rows of the
            // box: eight lanes per row (8 columns each), four rows per pass.
            if (box_in && write_w) {
              const int cc = lane & 7;
              const int jc = jb + cc * 8;
              __nv_bfloat16* wcol = static_cast<__nv_bfloat16*>(fd->w) + jc;
              uint4 wv[8], xv[8];
#pragma unroll
              for (int k = 0; k < 8; ++k) {   // all loads first
                const int rr = q * 32 + (lane >> 3) + 4 * k;
                const int ii = r0 + (lane >> 3) + 4 * k;
                xv[k] = *reinterpret_cast<const uint4*>(box + rr * 128 + ((cc ^ (rr & 7)) << 4));
                wv[k] = (ii < nrows && jc < ncols) ? *reinterpret_cast<const uint4*>(wcol + (int64_t)ii * fd->cols)
                                                   : make_uint4(0u, 0u, 0u, 0u);
              }
#pragma unroll
              for (int k = 0; k < 8; ++k) {
                const int ii = r0 + (lane >> 3) + 4 * k;
                if (ii >= nrows || jc >= ncols) continue;
                const uint32_t xw[4] = {xv[k].x, xv[k].y, xv[k].z, xv[k].w};
                uint32_t ww[4] = {wv[k].x, wv[k].y, wv[k].z, wv[k].w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const float w0 = bf_lo_w(ww[e]), w1 = bf_hi_w(ww[e]);
                  const float n0 = __fsub_rn(
                      w0, __fmul_rn(p.fuse.eM, __fadd_rn(__fmul_rn(fd->shape_scale, bf_lo_w(xw[e])),
                                                         __fmul_rn(p.fuse.lam, w0))));
                  const float n1 = __fsub_rn(
                      w1, __fmul_rn(p.fuse.eM, __fadd_rn(__fmul_rn(fd->shape_scale, bf_hi_w(xw[e])),
                                                         __fmul_rn(p.fuse.lam, w1))));
                  ww[e] = pack_bf2(n0, n1);
                }
                *reinterpret_cast<uint4*>(wcol + (int64_t)ii * fd->cols) = make_uint4(ww[0], ww[1], ww[2], ww[3]);
              }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&aux_empty[s]);   // the box's rows of this warp are read
          } else if (lane == 0) {
            if (box_in) {
              const TcGroupMaps& mp = p.maps[t.group];
              const CUtensorMap* dst = (phase == NS_GRAM) ? &mp.ast : (phase == NS_POLY ? &mp.bst : &mp.xst[cur ^ 1]);
              tma_store_3d(dst, box + q * 32 * 128, jb, r0, t.mat);
            }
            bulk_commit();
          }
        }
        if (stop) break;
        if (aux_phase && !fused && lane == 0) {
          // the slots go back to the aux loader once the stores have read them
          asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
          mbar_arrive(&aux_empty[2 * hw]);
          bulk_wait_read();
          mbar_arrive(&aux_empty[2 * hw + 1]);
        }
        __syncwarp();
      }
    }
    if (lane == 0) bulk_wait_all();
  }

  __syncwarp();
  pair_finish<kWStages>(*log, abort_flag, full, R.armed, rank);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemColsW);
  }
}

template <bool kMasked, bool kSplit, bool kGram>
cudaError_t set_attr_w() {
  return cudaFuncSetAttribute(ns_wide_kernel<kMasked, kSplit, kGram>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)WLayout<kGram>::kSmemBytes);
}

}  // namespace

cudaError_t launch_ns_wide(const TcParams& prm, int grid, bool masked, bool split, bool pdl, cudaStream_t st) {
  static bool attr_set[kMaxDevices] = {};
  const int slot = device_slot();
  if (slot < 0 || !attr_set[slot]) {
    cudaError_t e = set_attr_w<false, false, false>();
    if (e == cudaSuccess) e = set_attr_w<true, false, false>();
    if (e == cudaSuccess) e = set_attr_w<false, false, true>();
    if (e == cudaSuccess) e = set_attr_w<true, false, true>();
    if (e == cudaSuccess) e = set_attr_w<false, true, true>();
    if (e == cudaSuccess) e = set_attr_w<true, true, true>();
    if (e != cudaSuccess) return e;
    if (slot >= 0) attr_set[slot] = true;
  }
  count_launch();
  constexpr size_t sg = WLayout<true>::kSmemBytes, sa = WLayout<false>::kSmemBytes;
  if (prm.phase == NS_GRAM) {
    if (masked) {
      if (split) return launch_tc_kernel(ns_wide_kernel<true, true, true>, grid, sg, pdl, st, prm);
      return launch_tc_kernel(ns_wide_kernel<true, false, true>, grid, sg, pdl, st, prm);
    }
    if (split) return launch_tc_kernel(ns_wide_kernel<false, true, true>, grid, sg, pdl, st, prm);
    return launch_tc_kernel(ns_wide_kernel<false, false, true>, grid, sg, pdl, st, prm);
  }
  if (masked) return launch_tc_kernel(ns_wide_kernel<true, false, false>, grid, sa, pdl, st, prm);
  return launch_tc_kernel(ns_wide_kernel<false, false, false>, grid, sa, pdl, st, prm);
}

}  // namespace lm
