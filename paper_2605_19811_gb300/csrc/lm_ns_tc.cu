// Tensor-core Newton-Schulz phases for sm_103a: tcgen05.mma (bf16 operands,
// fp32 accumulators in TMEM) on CTA pairs (cta_group::2, one 256 x 256 tile
// per pair), operands staged by TMA into 128-byte-swizzled shared memory, a
// persistent grouped schedule over all same-shape matrices.
//
// Per NS iteration (Section 2, odd-polynomial Newton-Schulz), with the
// normalisation X / (||G_hat||_F + eps) folded into iteration 0.  A wide
// matrix (s x l, s <= l) iterates as
//   GRAM : A  = X X^T          K = l, only tiles on or above the diagonal
//   POLY : B  = b A + c A A    K = s, only tiles on or above the diagonal;
//                              the epilogue reads the A tile
//   APPLY: X' = a X + B X      K = s, all tiles; the epilogue reads the X tile
// and a tall one (l x s, kept in its own orientation) as A = X^T X and
// X' = a X + X B, which is the same function (p(X X^T) X = X p(X^T X)).
// A and A A are symmetric, so A A = A A^T and X B = X B^T: every operand is
// either K-major rows or MN-major columns of a stored matrix.
//
// A cluster of two CTAs computes one 256 x 256 tile: CTA r holds rows
// [128 r, 128 r + 128) of the A operand and N-rows [128 r, 128 r + 128) of the
// B operand, the pair's MMA (issued by CTA 0) leaves rows 128 r .. of the
// tile in CTA r's TMEM.  Each SM thus stages and reads half of B, which halves
// the shared-memory traffic per FLOP of a one-CTA 128 x 256 tile.
//
// CTA roles (352 threads, one CTA per SM):
//   warp 0    TMA producer (one elected lane), 5-stage smem ring (2 stages
//             of three-piece operands in the fp32 mode, see TcLayout); both CTAs'
//             copies signal CTA 0's full barrier
//   warp 1    TMEM allocator (both CTAs) + MMA issuer (CTA 0, one lane)
//   warps 2-9 epilogue: tcgen05.ld from TMEM, fused polynomial combination,
//             results written into shared memory (over the aux tile) and
//             stored by TMA, one 64-column box at a time.  Warps 2-5 (one
//             per TMEM lane quadrant and SM sub-partition) cover the whole
//             tile; warps 6-9 only work in a launch that also writes the
//             parameters, where each quadrant takes two warps, one per half
//             of the tile's columns (the W loads there are latency-bound).
//             Eight epilogue warps elsewhere measured 4% slower per Muon
//             step: two of them share each sub-partition's issue slots with
//             the producer or the MMA issuer.
//   warp 10   aux loader: TMA of the tile the POLY/APPLY epilogue combines
//             with the accumulator (A or X), issued while the main loop runs
// The last APPLY of a Muon step can also apply the parameter update
// W <- W - eta_M (s X_K + lambda W) (Algorithm 1, Muon branch) in its
// epilogue, and X_K itself is never stored.  Where a is folded into B' (the
// default), the aux loader brings the W tile by TMA, the epilogue updates it
// in shared memory from the accumulator and stores it back by TMA (W tensor
// maps per matrix in global memory).  Otherwise the aux tile is X, X_K goes
// to shared memory as bf16, and each warp then reads its 32 rows of W with
// coalesced 16-byte loads, updates and writes them.
// Tiles are assigned to pairs on the host by a longest-first greedy balance
// of their K lengths (a contiguous range per pair).
// kAccBufs 256-column accumulators in TMEM (two let the epilogue of one tile
// overlap the main loop of the next).  Every mbarrier wait is bounded in time; a wait that
// gives up sets LM_FLAG_TIMEOUT, makes the other roles stop, waits (bounded)
// for its own copies and MMAs, frees TMEM and returns.
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include "lm_ns_tc_shared.cuh"

namespace lm {
namespace {

using namespace tc;    // PTX wrappers (lm_tc_ptx.cuh)
using namespace tcs;   // constants, stop check and end-of-launch handshake (lm_ns_tc_shared.cuh)

constexpr int kAccBufs = 2;                          // 256-column accumulators in TMEM
constexpr int kFuseBatch = 4;   // W loads in flight per thread in the global-memory parameter write
constexpr int kTmemCols = kAccBufs * BN;
// Shared-memory layout per operand precision.  kP = 1: bf16 operands, a
// 5-stage ring of 32 KB per CTA and a 64 KB aux/staging buffer.  kP = 3:
// fp32 operands held as three bf16 pieces (hi + mid + lo, exact), a 2-stage
// ring of 96 KB per CTA and a 4 KB transpose tile per epilogue warp (that
// epilogue reads its aux values and writes its results through global memory).
template <int kP>
struct TcLayout {
  static constexpr int kStages = kP == 1 ? 5 : 2;
  static constexpr int kStageBytes = kP * (kABytes + kBBytes);
  static constexpr size_t kAuxOffset = (size_t)kStages * kStageBytes;
  // kP = 1: the aux / staging boxes; kP = 3: a 32 x 33 fp32 transpose tile per epilogue warp
  static constexpr size_t kBarOffset = kAuxOffset + (kP == 1 ? 4 * kAuxBoxBytes : 8 * 32 * 33 * 4);
  static constexpr size_t kSmemBytes = 1024 /*align slack*/ + kBarOffset + 256;
};

// Operands of one tile.  Wide groups hold X as s x l, tall groups as l x s
// (the parameter's own orientation):
//   GRAM  wide: A = X X^T, both operands K-major rows of X (K = l)
//         tall: A = X^T X, both operands MN-major columns of X (K = l)
//   POLY      : B = b A + c A A, operands rows of A (K = s)
//   APPLY wide: X' = a X + B X, rows of B and MN-major X (K = s)
//         tall: X' = a X + X B, K-major rows of X and rows of B (K = s)
// A and B are symmetric and only their 256 x 256 tiles on or above the
// diagonal are stored.  A row block r of A (or B) therefore reads K blocks
// k >= 256 r K-major from the stored tiles, and K blocks below 256 r as the
// transposed stored tile, i.e. MN-major.  The split falls on a 256 boundary,
// so both CTAs of a pair use the same layout for every K block.
struct OpSeg {
  int kb_end;                    // K blocks [previous end, kb_end)
  bool a_mn, b_mn;
  const CUtensorMap* map_a;
  const CUtensorMap* map_b;
};
struct TilePlan {
  int nseg;
  int nk;
  int kb_start;   // first K block (split Gram tiles start inside K)
  OpSeg seg[3];
};
__device__ __forceinline__ void plan_push(TilePlan& P, int kb_end, bool a_mn, bool b_mn,
                                          const CUtensorMap* ma, const CUtensorMap* mb) {
  const int prev = P.nseg ? P.seg[P.nseg - 1].kb_end : 0;
  if (kb_end <= prev) return;    // empty range
  P.seg[P.nseg++] = OpSeg{kb_end, a_mn, b_mn, ma, mb};
}
__device__ __forceinline__ TilePlan tile_plan(int phase, const NsGroup& g, const TcGroupMaps& mp, int cur,
                                              const NsTile& t, bool from_a = false) {
  TilePlan P;
  P.nseg = 0;
  P.kb_start = 0;
  if (phase == NS_GRAM) {
    P.nk = g.l_pad / BK;
    const int kb_end = t.kb1 != 0 ? (int)t.kb1 : P.nk;
    P.kb_start = t.kb1 != 0 ? (int)t.kb0 : 0;
    if (g.tall) plan_push(P, kb_end, true, true, &mp.xmn[cur], &mp.xmn[cur]);
    else plan_push(P, kb_end, false, false, &mp.xk[cur], &mp.xk[cur]);
    return P;
  }
  P.nk = g.s_pad / BK;
  const int ka = min(t.tm * (BM / BK), P.nk);   // first K block on or above row block tm
  const int kn = min(t.tn * (BN / BK), P.nk);   // the same for column block tn
  if (phase == NS_POLY) {            // A-operand rows tm, B-operand rows tn (tn >= tm)
    plan_push(P, ka, true, true, &mp.amn, &mp.amn);
    plan_push(P, kn, false, true, &mp.a, &mp.amn);
    plan_push(P, P.nk, false, false, &mp.a, &mp.a);
    return P;
  }
  // APPLY: the left operand is B, or A where B = b A was not formed (the
  // same upper-tile storage)
  const CUtensorMap* lmn = from_a ? &mp.amn : &mp.bmn;
  const CUtensorMap* lk = from_a ? &mp.a : &mp.b;
  if (!g.tall) {                     // rows tm of B, X MN-major
    plan_push(P, ka, true, true, lmn, &mp.xmn[cur]);
    plan_push(P, P.nk, false, true, lk, &mp.xmn[cur]);
  } else {                           // rows of X K-major, rows tn of B
    plan_push(P, kn, false, true, &mp.xk[cur], lmn);
    plan_push(P, P.nk, false, false, &mp.xk[cur], lk);
  }
  return P;
}


// Producer k-loop of one tile, specialised on the operand layouts (a loop
// with per-block layout branches measured ~12% slower end to end).
// K-major operand half: one 64 (K) x 128 box; MN-major: one 4-D box that
// fills both 64 (MN) x 64 (K) swizzle atoms (one copy instead of two
// measured ~2% faster).  Returns false if a wait gave up.
template <int kS>
struct ProducerRing {
  int stage;
  uint32_t ph;
  int armed[kS];
};
// kP pieces per operand: piece q of matrix mat is matrix mat + q * pstride
// of the tensor map; a stage holds the kP A pieces, then the kP B pieces.
// same: both operands are the same rows of the same matrix (a diagonal Gram
// or polynomial tile), so only the A boxes are loaded and the MMA reads them
// as B too.
template <bool AMN, bool BMN, int kP>
__device__ __forceinline__ bool produce_range(ProducerRing<TcLayout<kP>::kStages>& R,
                                              ProducerLog<TcLayout<kP>::kStages>& log, uint8_t* smem,
                                              uint64_t* full, uint64_t* empty, volatile int* abort_flag,
                                              uint64_t wait_ns, uint32_t rank, int kb0, int kb1,
                                              const CUtensorMap* map_a, const CUtensorMap* map_b, int row_a,
                                              int col_b, int mat, int pstride, bool same) {
  using L = TcLayout<kP>;
  const uint32_t own = same ? (uint32_t)(kP * kABytes) : (uint32_t)L::kStageBytes;   // this CTA's bytes
  for (int kb = kb0; kb < kb1; ++kb) {
    if (!mbar_wait(&empty[R.stage], R.ph ^ 1u, abort_flag, wait_ns)) return false;
    uint8_t* sa = smem + (size_t)R.stage * L::kStageBytes;
    uint8_t* sb = sa + kP * kABytes;
    const uint32_t fb = peer_addr(&full[R.stage], 0);
    if (rank == 0) {
      mbar_arrive_expect_tx(&full[R.stage], 2u * own);
      R.armed[R.stage] = (int)R.ph;
    }
    log.bytes[R.stage] = own;
    log.n += 1u;
    const int k0 = kb * BK;
#pragma unroll
    for (int q = 0; q < kP; ++q) {
      if (!AMN) tma_load_3d(sa + q * kABytes, map_a, fb, k0, row_a, mat + q * pstride);
      else tma_load_4d(sa + q * kABytes, map_a, fb, 0, k0, row_a >> 6, mat + q * pstride);
    }
#pragma unroll
    for (int q = 0; q < kP && !same; ++q) {
      if (!BMN) tma_load_3d(sb + q * kBBytes, map_b, fb, k0, col_b, mat + q * pstride);
      else tma_load_4d(sb + q * kBBytes, map_b, fb, 0, k0, col_b >> 6, mat + q * pstride);
    }
    if (++R.stage == L::kStages) {
      R.stage = 0;
      R.ph ^= 1u;
    }
  }
  return true;
}

// MMA issue for K blocks [kb0, kb1) of one tile with fixed operand layouts.
// kP = 3: with A = A0 + A1 + A2 and B = B0 + B1 + B2 (each piece 2^-8 of the
// previous in magnitude) the six products of order up to 2^-16 are summed,
// A0B0 + A0B1 + A1B0 + A0B2 + A2B0 + A1B1; the dropped ones are of order 2^-24.
// A0B0 goes into the accumulator d_tmem and the five smaller products into
// d_cross; the epilogue adds the two in fp32.  The tensor cores' fp32
// accumulation loses about one unit of the last place of the accumulator per
// MMA, in the same direction (measured: the error grows with the number of
// MMAs summed, 2.2e-5 relative for a 1280-deep product with all six in one
// accumulator), so the large accumulator takes a sixth of the additions and
// the errors of the other are 2^-8 smaller.
template <bool AMN, bool BMN, int kP>
__device__ __forceinline__ bool mma_range(int& stage, uint32_t& ph, uint8_t* smem, uint64_t* full,
                                          uint64_t* empty, volatile int* abort_flag, uint64_t wait_ns, int kb0,
                                          int kb1, uint32_t d_tmem, uint32_t d_cross, int kb_first, bool same) {
  using L = TcLayout<kP>;
  constexpr int kProducts = kP == 1 ? 1 : 6;
  constexpr int qa[6] = {0, 0, 1, 0, 2, 1};
  constexpr int qb[6] = {0, 1, 0, 2, 0, 1};
  const uint32_t idesc = make_idesc(BM, BN, AMN, BMN);
  for (int kb = kb0; kb < kb1; ++kb) {
    if (!mbar_wait(&full[stage], ph, abort_flag, wait_ns)) return false;
    tc_fence_after();
    const uint32_t sa = smem_u32(smem + (size_t)stage * L::kStageBytes);
    const uint32_t sb = same ? sa : sa + kP * kABytes;   // kBBytes == kABytes
    // descriptors of the stage's K = 0 slices; a 16-deep K step adds its
    // byte offset / 16 to the start-address field (bits 0-13: no carry, the
    // shared-memory window is below 2^18 bytes)
    const uint64_t a0 = AMN ? sw128_desc(sa, 64 * BK * 2, 1024) : sw128_desc(sa, 16, 1024);
    const uint64_t b0 = BMN ? sw128_desc(sb, 64 * BK * 2, 1024) : sw128_desc(sb, 16, 1024);
#pragma unroll
    for (int kk = 0; kk < BK / 16; ++kk) {
#pragma unroll
      for (int m = 0; m < kProducts; ++m) {
        const uint64_t adesc = a0 + (uint64_t)((qa[m] * kABytes + kk * (AMN ? 2048 : 32)) >> 4);
        const uint64_t bdesc = b0 + (uint64_t)((qb[m] * kBBytes + kk * (BMN ? 2048 : 32)) >> 4);
        const bool first = kb == kb_first && kk == 0 && m <= 1;   // first product into each accumulator
        umma_bf16(m == 0 ? d_tmem : d_cross, adesc, bdesc, idesc, first ? 0u : 1u);
      }
    }
    umma_commit_pair(&empty[stage]);
    if (++stage == L::kStages) {
      stage = 0;
      ph ^= 1u;
    }
  }
  return true;
}

// fp32 value v as hi + mid + lo bf16 pieces, exactly: each piece takes the
// next 8 significant bits (the differences are exact in fp32).
__device__ __forceinline__ void split3(float v, float& h, float& m, float& l) {
  h = __bfloat162float(__float2bfloat16_rn(v));
  const float r1 = v - h;
  m = __bfloat162float(__float2bfloat16_rn(r1));
  l = r1 - m;
}
// Epilogue of one 32 x 32 chunk (rows r0 .. r0 + 31, one per lane; columns
// j0 ..) with three-piece operands; aux values and results go through global
// memory, coalesced through the warp's transpose tile stg: lane l reads and
// writes 16 bytes of row l / 4 + 8 k (k = 0 .. 3), so a warp access covers 8
// rows x 64 bytes of one plane.
//   kacc: APPLY's factor on the accumulator (1, or b where B = b A was not
//   formed).
//   aux: the A (POLY) or X (APPLY) element, hi + mid + lo; out: the result's
//   pieces, or fp32 in out_f32 (last APPLY).  base: element (r0, j0) of the
//   matrix in plane 0; ld: row length; plane: elements per piece.
__device__ __forceinline__ void piece_chunk(const uint32_t (&r)[32], int phase, const NsCoeffs& co, float nscale,
                                            float kacc,
                                            const __nv_bfloat16* aux, __nv_bfloat16* out, float* out_f32,
                                            size_t plane, size_t base, size_t ld, bool row_ok, int j0, int ncols,
                                            float (*stg)[33], int lane) {
  const int rr = lane >> 2, c8 = (lane & 3) * 8;
  float v[32];
  if (phase != NS_GRAM) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int row = rr + 8 * k;
      float a8[8];
#pragma unroll
      for (int t = 0; t < 8; ++t) a8[t] = 0.f;
#pragma unroll
      for (int q = 0; q < 3; ++q) {
        const uint4 a4 = *reinterpret_cast<const uint4*>(aux + q * plane + base + (size_t)row * ld + c8);
        const uint32_t aw[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          a8[2 * e] += bf_lo(aw[e]);
          a8[2 * e + 1] += bf_hi(aw[e]);
        }
      }
#pragma unroll
      for (int t = 0; t < 8; ++t) stg[row][c8 + t] = a8[t];
    }
    __syncwarp();
#pragma unroll
    for (int e = 0; e < 32; ++e) v[e] = stg[lane][e];
    __syncwarp();
  }
#pragma unroll
  for (int e = 0; e < 32; ++e) {
    const float acc = __uint_as_float(r[e]);
    float o;
    if (phase == NS_GRAM) o = acc * nscale;
    else if (phase == NS_POLY) o = co.b * v[e] + co.c * acc;
    else o = __fmaf_rn(co.a, v[e], kacc * acc) * nscale;   // kacc = 1: exactly a v + acc, one rounding
    stg[lane][e] = (row_ok && j0 + e < ncols) ? o : 0.f;
  }
  __syncwarp();
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int row = rr + 8 * k;
    float o8[8];
#pragma unroll
    for (int t = 0; t < 8; ++t) o8[t] = stg[row][c8 + t];
    const size_t off = base + (size_t)row * ld + c8;
    if (out_f32 != nullptr) {
      float4* dst = reinterpret_cast<float4*>(out_f32 + off);
      dst[0] = make_float4(o8[0], o8[1], o8[2], o8[3]);
      dst[1] = make_float4(o8[4], o8[5], o8[6], o8[7]);
      continue;
    }
    uint32_t w[3][4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      float h0, m0, l0, h1, m1, l1;
      split3(o8[2 * e], h0, m0, l0);
      split3(o8[2 * e + 1], h1, m1, l1);
      w[0][e] = pack_bf2(h0, h1);
      w[1][e] = pack_bf2(m0, m1);
      w[2][e] = pack_bf2(l0, l1);
    }
#pragma unroll
    for (int q = 0; q < 3; ++q)
      *reinterpret_cast<uint4*>(out + q * plane + off) = make_uint4(w[q][0], w[q][1], w[q][2], w[q][3]);
  }
  __syncwarp();   // the tile is reused by the next chunk
}

// ------------------------------- the kernel ---------------------------------
// kMasked: the launch carries a per-matrix mask (stable-rank selection);
// kSplit: its Gram tiles include split-K parts.  The plain instantiation keeps
// the common path free of both.  kP: bf16 pieces per operand value (1: bf16
// operands; 3: fp32 operands as hi + mid + lo bf16 pieces, six products).
template <bool kMasked, bool kSplit, int kP>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    ns_tc_kernel(const __grid_constant__ TcParams p) {
  using L = TcLayout<kP>;
  constexpr int kStages = L::kStages;
  // tiles in flight in TMEM: kP = 1 double-buffers two accumulators; kP = 3
  // gives one tile both (main and cross products)
  constexpr int kAccRing = kP == 1 ? kAccBufs : 1;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* auxbuf = smem + L::kAuxOffset;   // kP = 1: 4 x (128 rows x 64 cols) bf16, 128-byte swizzled
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L::kBarOffset);
  uint64_t* empty = full + kStages;
  uint64_t* accfull = empty + kStages;
  uint64_t* accempty = accfull + 2;
  uint64_t* aux_full = accempty + 2;
  uint64_t* aux_empty = aux_full + 1;
  uint64_t* done = aux_empty + 1;
  ProducerLog<kStages>* log = reinterpret_cast<ProducerLog<kStages>*>(done + 1);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(log + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint32_t* stop_word = tmem_slot + 2;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int phase = p.phase;
  const int cur = p.iter & 1;
  const uint32_t rank = cluster_rank();          // 0: MMA issuer of the pair
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  // epilogue reads the A (POLY) or X (APPLY) tile; an APPLY whose B has a
  // folded into its diagonal needs no X tile
  // The last APPLY of a Muon step may also write the parameters.  Where a is
  // folded into B' its aux tile is the W tile, updated in shared memory and
  // stored back by TMA; otherwise the aux tile is X and W is read from global
  // memory after the tile (eight epilogue warps for the latency).
  const bool fused_launch = phase == NS_APPLY && p.fuse.mats != nullptr;
  const bool fuse_w_tile = kP == 1 && fused_launch && p.fold_a;
  const bool aux_phase = kP == 1 && phase != NS_GRAM && (!(phase == NS_APPLY && p.fold_a) || fuse_w_tile);
  // Active epilogue warps: one per TMEM lane quadrant (and SM sub-partition)
  // except in a parameter write that reads W from global memory.
  const int nepi = (kP == 1 && !(fused_launch && !fuse_w_tile)) ? 4 : kEpiWarps;
  // this pair's tiles: a host-balanced range, or round robin
  int w_begin = p.offsets ? p.offsets[pair] : pair;
  const int w_end = p.offsets ? p.offsets[pair + 1] : p.ntiles;
  const int w_step = p.offsets ? 1 : npairs;

  if constexpr (kMasked) {
    // A pair none of whose tiles belongs to a selected matrix leaves before
    // any barrier, TMEM or cluster work (the roles would otherwise walk its
    // tile list one dependent load chain at a time).  Both CTAs of the pair
    // scan the same range of the same mask, so both leave or both stay.  The
    // mask comes from a kernel this launch may overlap: wait for it first.
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
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < kAccBufs; ++b) {
      mbar_init(&accfull[b], 1);
      mbar_init(&accempty[b], 2 * nepi);
    }
    mbar_init(aux_full, 1);
    mbar_init(aux_empty, nepi);
    mbar_init(done, 1);
    log->n = 0;
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  if (pair_start(p, stop_word, rank)) w_begin = w_end;   // an earlier launch gave up: no tiles
  const uint32_t tmem_base = *tmem_slot;
  const uint64_t wait_ns = p.wait_ns;

  auto give_up = [&]() {
    *abort_flag = 1;
    atomicOr(p.flags, LM_FLAG_TIMEOUT);
  };

  ProducerRing<kStages> R;   // producer lane: ring position and armed phases
  R.stage = 0;
  R.ph = 0;
  for (int s = 0; s < kStages; ++s) R.armed[s] = -1;

  if (warp == 0) {
    // ------------------------------ producer ------------------------------
    if (lane == 0) {
      bool ok = true;
      // the next tile's entry is loaded one tile ahead (its latency then
      // falls inside the current tile, not between two tiles' MMAs)
      NsTile tnext = w_begin < w_end ? p.tiles[w_begin] : NsTile{};
      for (int w = w_begin; ok && w < w_end; w += w_step) {
        const NsTile t = tnext;
        if (w + w_step < w_end) tnext = p.tiles[w + w_step];
        if (kMasked && !tile_active(p, t)) continue;
        const NsGroup& g = p.groups[t.group];
        const TilePlan P = tile_plan(phase, g, p.maps[t.group], cur, t, p.apply_from_a != 0);
        const int row_a = t.tm * BM + (int)rank * kHalf;
        const int col_b = t.tn * BN + (int)rank * kHalf;
        int kb0 = P.kb_start;
        for (int sg = 0; ok && sg < P.nseg; ++sg) {
          const OpSeg& S = P.seg[sg];
          if (!S.a_mn && !S.b_mn)
            ok = produce_range<false, false, kP>(R, *log, smem, full, empty, abort_flag, wait_ns, rank, kb0, S.kb_end, S.map_a,
                                             S.map_b, row_a, col_b, t.mat, g.count,
                                             S.map_a == S.map_b && row_a == col_b);
          else if (!S.a_mn)
            ok = produce_range<false, true, kP>(R, *log, smem, full, empty, abort_flag, wait_ns, rank, kb0, S.kb_end, S.map_a,
                                            S.map_b, row_a, col_b, t.mat, g.count,
                                             S.map_a == S.map_b && row_a == col_b);
          else
            ok = produce_range<true, true, kP>(R, *log, smem, full, empty, abort_flag, wait_ns, rank, kb0, S.kb_end, S.map_a,
                                           S.map_b, row_a, col_b, t.mat, g.count,
                                             S.map_a == S.map_b && row_a == col_b);
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
      int ab = 0;
      uint32_t aph = 0;
      bool ok = true;
      // the next tile's entry is loaded one tile ahead (its latency then
      // falls inside the current tile, not between two tiles' MMAs)
      NsTile tnext = w_begin < w_end ? p.tiles[w_begin] : NsTile{};
      for (int w = w_begin; ok && w < w_end; w += w_step) {
        const NsTile t = tnext;
        if (w + w_step < w_end) tnext = p.tiles[w + w_step];
        if (kMasked && !tile_active(p, t)) continue;
        const NsGroup& g = p.groups[t.group];
        const TilePlan P = tile_plan(phase, g, p.maps[t.group], cur, t, p.apply_from_a != 0);
        if (!mbar_wait(&accempty[ab], aph ^ 1u, abort_flag, wait_ns)) {
          give_up();
          break;
        }
        tc_fence_after();
        // kP = 1: accumulator ab; kP = 3: the main products in the first 256
        // columns, the cross products in the second
        const uint32_t d_tmem = tmem_base + (uint32_t)(ab * BN);
        const uint32_t d_cross = tmem_base + (uint32_t)BN;
        int kb0 = P.kb_start;
        for (int sg = 0; ok && sg < P.nseg; ++sg) {
          const OpSeg& S = P.seg[sg];
          if (!S.a_mn && !S.b_mn)
            ok = mma_range<false, false, kP>(stage, ph, smem, full, empty, abort_flag, wait_ns, kb0, S.kb_end, d_tmem, d_cross,
                                            P.kb_start, S.map_a == S.map_b && t.tm == t.tn);
          else if (!S.a_mn)
            ok = mma_range<false, true, kP>(stage, ph, smem, full, empty, abort_flag, wait_ns, kb0, S.kb_end, d_tmem, d_cross,
                                            P.kb_start, S.map_a == S.map_b && t.tm == t.tn);
          else
            ok = mma_range<true, true, kP>(stage, ph, smem, full, empty, abort_flag, wait_ns, kb0, S.kb_end, d_tmem, d_cross,
                                            P.kb_start, S.map_a == S.map_b && t.tm == t.tn);
          kb0 = S.kb_end;
        }
        if (!ok) give_up();
        if (!ok) break;
        umma_commit_pair(&accfull[ab]);
        if (++ab == kAccRing) {
          ab = 0;
          aph ^= 1u;
        }
      }
      // all issued MMAs complete before TMEM is released
      umma_commit_local(done);
      volatile int never = 0;
      mbar_wait(done, 0, &never, kCleanupWaitNs);
    }
  } else if (warp == kAuxWarp) {
    // --------------------------- aux tile loader ---------------------------
    // The epilogue of POLY needs the A tile, that of APPLY the X tile (or the
    // W tile of a parameter write); each is loaded by TMA into auxbuf while
    // the tile's main loop runs.  W boxes past the parameter's extent read
    // zeros.
    if (lane == 0 && aux_phase) {
      uint32_t xph = 0;
      int armed = -1;
      bool ok = true;
      for (int w = w_begin; ok && w < w_end; w += w_step) {
        const NsTile t = p.tiles[w];
        if (kMasked && !tile_active(p, t)) continue;
        const TcGroupMaps& mp = p.maps[t.group];
        const CUtensorMap* map = (phase == NS_POLY) ? &mp.a : &mp.xk[cur];
        int zc = t.mat;
        if (fuse_w_tile) {   // the W load map of this matrix (two maps per matrix: load, store)
          map = p.fuse.wmaps + 2 * (p.groups[t.group].first_mat + t.mat);
          zc = 0;
        }
        if (!mbar_wait(aux_empty, xph ^ 1u, abort_flag, wait_ns)) {
          give_up();
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(aux_full, 4 * kAuxBoxBytes);
        armed = (int)xph;
        const int row0 = t.tm * BM + (int)rank * kHalf;
#pragma unroll
        for (int b = 0; b < 4; ++b)
          tma_load_3d_local(auxbuf + b * kAuxBoxBytes, map, aux_full, t.tn * BN + 64 * b, row0, zc);
        xph ^= 1u;
      }
      if (!ok && armed >= 0) {
        volatile int never = 0;
        mbar_wait(aux_full, (uint32_t)armed, &never, kCleanupWaitNs);
      }
    }
  } else {
    // ------------------------------ epilogue -------------------------------
    // Thread (quadrant q, lane) owns one row of this CTA's half tile and
    // 128 (nepi = 8) or all 256 (nepi = 4) of its columns, in 32-column chunks.
    // Results go into auxbuf (over the aux values, if any) in the 128-byte
    // swizzled box layout and leave by TMA stores, 32 rows x 64 columns each.
    // A warp stores each 64-column box as soon as its two chunks are written
    // rather than both boxes at the end of the tile: all pairs run tiles of
    // equal length, so stores issued at tile end coincide across the GPU and
    // starve the operand loads (measured: 2846 -> 1568 cycles per APPLY tile
    // of the MMA issuer waiting for operands; APPLY 2% faster).
    const int q = warp & 3;                   // TMEM lane quadrant of this warp
    const int half0 = nepi == 8 ? (warp - 2) >> 2 : 0;   // first 128 columns of the tile it covers
    const int nhalves = 8 / nepi;
    const int row = q * 32 + lane;            // row of this CTA's half tile
    const uint32_t acc_empty0 = peer_addr(&accempty[0], 0);
    const uint32_t acc_empty1 = peer_addr(&accempty[kAccRing - 1], 0);
    int ab = 0;
    uint32_t aph = 0, xph = 0;
    for (int w = (warp - 2 < nepi) ? w_begin : w_end; w < w_end; w += w_step) {
      const NsTile t = p.tiles[w];
      if (kMasked && !tile_active(p, t)) continue;
      const NsGroup& g = p.groups[t.group];
      const bool fused = phase == NS_APPLY && p.fuse.mats != nullptr;
      const MatDesc* fd = fused ? &p.fuse.mats[g.first_mat + t.mat] : nullptr;
      // a tile whose epilogue starts after a give-up was recorded leaves W alone
      const unsigned flags_now = fused && lane == 0 ? *reinterpret_cast<volatile unsigned*>(p.flags) : 0u;
      const bool write_w = fused && __shfl_sync(0xffffffffu, flags_now, 0) == 0u;
      bool ok = true;
      if (lane == 0) {
        ok = mbar_wait(&accfull[ab], aph, abort_flag, wait_ns);
        if (ok && aux_phase) ok = mbar_wait(aux_full, xph, abort_flag, wait_ns);
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      if (!ok) {
        if (lane == 0) give_up();
        break;
      }
      tc_fence_after();

      // APPLY: X' = a X + B X, or a X + b (A X) where B = b A was not formed
      const float kacc = p.apply_from_a ? p.co.b : 1.f;
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
      const int i = r0 + lane;
      const bool warp_in = r0 < row_lim;        // rows past the padded matrix are skipped
      const bool split = kSplit && phase == NS_GRAM && t.slot != 0;
      if (fused && lane == 0 && q == 0 && half0 == 0 && rank == 0 && t.tm == 0 && t.tn == 0 &&
          !isfinite((float)sqrt(p.norm2[g.first_mat + t.mat])))
        atomicOr(p.flags, LM_FLAG_NONFINITE);
      for (int c4 = 0; c4 < 4 * nhalves; ++c4) {
        const int ch = half0 * 4 + c4;
        uint32_t r[32];
        __syncwarp();   // tcgen05.ld is warp-collective: reconverge first
        tmem_ld32(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * BN + ch * 32), r);
        if (kP == 3) {   // main + cross accumulators
          uint32_t rc[32];
          tmem_ld32(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(BN + ch * 32), rc);
#pragma unroll
          for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) + __uint_as_float(rc[e]));
        }
        const int j0 = t.tn * BN + ch * 32;
        if (!warp_in || j0 >= jmax) continue;   // beyond the padded matrix
        if (kP == 3 && !split) {
          // rows of the output: s_pad or l_pad (APPLY tall); ld its row length
          const size_t ld = (size_t)(phase == NS_APPLY ? (g.tall ? g.s_pad : g.l_pad) : g.s_pad);
          const size_t msize = (size_t)(phase == NS_APPLY ? (size_t)g.s_pad * g.l_pad : (size_t)g.s_pad * g.s_pad);
          const size_t base = (size_t)t.mat * msize + (size_t)r0 * ld + j0;   // row r0 = this warp's first
          const size_t plane = (size_t)g.count * msize;
          const __nv_bfloat16* aux = static_cast<const __nv_bfloat16*>(phase == NS_POLY ? g.A : g.X[cur]);
          __nv_bfloat16* out = static_cast<__nv_bfloat16*>(phase == NS_GRAM ? g.A : (phase == NS_POLY ? g.B : g.X[cur ^ 1]));
          float* out_f32 = (phase == NS_APPLY && p.final_f32) ? static_cast<float*>(g.Xf) : nullptr;
          float (*stg)[33] = reinterpret_cast<float (*)[33]>(auxbuf) + (warp - 2) * 32;
          piece_chunk(r, phase, p.co, nscale, kacc, aux, out, out_f32, plane, base, ld, i < nrows, j0, ncols, stg,
                      lane);
          continue;
        }
        if (split) {
          // partial Gram product of a split tile: its own fp32 workspace tile
          float* wrow = p.split_ws + (size_t)(t.slot - 1) * (BM * BN) + (size_t)((int)rank * kHalf + row) * BN +
                        ch * 32;
#pragma unroll
          for (int e = 0; e < 32; e += 4) {
            float o[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const int j = j0 + e + u;
              o[u] = (i < nrows && j < ncols) ? __uint_as_float(r[e + u]) * nscale : 0.f;
            }
            *reinterpret_cast<float4*>(wrow + e) = make_float4(o[0], o[1], o[2], o[3]);
          }
          continue;
        }
        // 16-byte chunk c of row r of a box sits at chunk position c ^ (r mod 8)
        uint4* abox = reinterpret_cast<uint4*>(auxbuf + (ch >> 1) * kAuxBoxBytes + row * 128);
        const int csub = (ch & 1) * 4;
        float v[32];
        if (aux_phase) {
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const uint4 a4 = abox[(csub + u) ^ (row & 7)];
            const uint32_t aw[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              v[u * 8 + 2 * e] = bf_lo(aw[e]);
              v[u * 8 + 2 * e + 1] = bf_hi(aw[e]);
            }
          }
        }
        // One loop per phase (the branches are uniform), and the padding mask
        // only on chunks that reach past the true extent: the element loop with
        // all of them inside measured 2% slower per Muon step (issue slots
        // shared with the producer and MMA-issuer warps).
        if (fuse_w_tile) {
          // W <- W - eta_M (s X_K + lambda W) (Algorithm 1, Muon branch) on
          // the W tile, with X_K = B' X rounded to bf16 as it would have been
          // stored; entries past W's extent are not stored (TMA clips them)
          const float ss = fd->shape_scale;
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const float xk = __bfloat162float(__float2bfloat16_rn(__uint_as_float(r[e]) * nscale));
            const float wo = v[e];
            v[e] = __fsub_rn(wo, __fmul_rn(p.fuse.eM, __fadd_rn(__fmul_rn(ss, xk), __fmul_rn(p.fuse.lam, wo))));
          }
        } else if (phase == NS_POLY) {
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] = p.co.b * v[e] + p.co.c * __uint_as_float(r[e]);
          if (p.fold_a && t.tm == t.tn) {   // B' = a I + B
#pragma unroll
            for (int e = 0; e < 32; ++e)
              if (i == j0 + e) v[e] += p.co.a;
          }
        } else if (phase == NS_APPLY && !p.fold_a) {
#pragma unroll
          for (int e = 0; e < 32; ++e)
            v[e] = __fmaf_rn(p.co.a, v[e], kacc * __uint_as_float(r[e])) * nscale;   // the same rounding as ns_wide_kernel
        } else if (nscale != 1.f) {          // GRAM, or X' = B' X
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] = __uint_as_float(r[e]) * nscale;
        } else {
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] = __uint_as_float(r[e]);
        }
        if (!fuse_w_tile && (i >= nrows || j0 + 32 > ncols)) {   // padding outside the true extent stays zero
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] = (i < nrows && j0 + e < ncols) ? v[e] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u)
          abox[(csub + u) ^ (row & 7)] =
              make_uint4(pack_bf2(v[u * 8 + 0], v[u * 8 + 1]), pack_bf2(v[u * 8 + 2], v[u * 8 + 3]),
                         pack_bf2(v[u * 8 + 4], v[u * 8 + 5]), pack_bf2(v[u * 8 + 6], v[u * 8 + 7]));
        if (kP == 1 && (!fused || fuse_w_tile) && (c4 & 1)) {
          // box ch / 2 of this warp's 32 rows is complete: store it now (a
          // parameter write stores W boxes that reach into W, unless a wait
          // of this step gave up)
          fence_proxy_async_smem();
          __syncwarp();
          const int b = ch >> 1;
          const int x0 = t.tn * BN + 64 * b;
          if (lane == 0 && (!fused || (write_w && x0 < fd->cols && r0 < fd->rows))) {
            const TcGroupMaps& mp = p.maps[t.group];
            const CUtensorMap* dst = (phase == NS_GRAM) ? &mp.ast : (phase == NS_POLY ? &mp.bst : &mp.xst[cur ^ 1]);
            if (fused) dst = p.fuse.wmaps + 2 * (g.first_mat + t.mat) + 1;
            tma_store_3d(dst, auxbuf + b * kAuxBoxBytes + q * 32 * 128, x0, r0, fused ? 0 : t.mat);
            bulk_commit();
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(ab == 0 ? acc_empty0 : acc_empty1);
      if (++ab == kAccRing) {
        ab = 0;
        aph ^= 1u;
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (fused && !fuse_w_tile) {
        // Last APPLY: W <- W - eta_M (s X_K + lambda W), with X_K the bf16
        // values just written to auxbuf.  Half-warp h covers row 2k + h of the
        // warp's 32 rows, 16 lanes x 8 columns = 256 contiguous bytes of W.
        for (int half = half0; half < half0 + nhalves; ++half) {
          if (warp_in && write_w) {
            const int cc = lane & 15;
            const int jc = t.tn * BN + half * 128 + cc * 8;
            const unsigned char* box = auxbuf + (2 * half + (cc >> 3)) * kAuxBoxBytes;
            const int ibase = t.tm * BM + (int)rank * kHalf + q * 32 + (lane >> 4);
            __nv_bfloat16* wcol = static_cast<__nv_bfloat16*>(fd->w) + jc;
            for (int k0 = 0; k0 < 16; k0 += kFuseBatch) {
              uint4 wv[kFuseBatch], xv[kFuseBatch];
#pragma unroll
              for (int u = 0; u < kFuseBatch; ++u) {   // all loads of the batch first
                const int rr = q * 32 + 2 * (k0 + u) + (lane >> 4);
                const int ii = ibase + 2 * (k0 + u);
                xv[u] = *reinterpret_cast<const uint4*>(box + rr * 128 + (((cc & 7) ^ (rr & 7)) << 4));
                wv[u] = (ii < nrows && jc < ncols)
                            ? *reinterpret_cast<const uint4*>(wcol + (int64_t)ii * fd->cols)
                            : make_uint4(0u, 0u, 0u, 0u);
              }
#pragma unroll
              for (int u = 0; u < kFuseBatch; ++u) {
                const int ii = ibase + 2 * (k0 + u);
                if (ii >= nrows || jc >= ncols) continue;
                const uint32_t xw[4] = {xv[u].x, xv[u].y, xv[u].z, xv[u].w};
                uint32_t ww[4] = {wv[u].x, wv[u].y, wv[u].z, wv[u].w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const float w0 = bf_lo(ww[e]), w1 = bf_hi(ww[e]);
                  const float n0 = __fsub_rn(w0, __fmul_rn(p.fuse.eM, __fadd_rn(__fmul_rn(fd->shape_scale, bf_lo(xw[e])),
                                                                               __fmul_rn(p.fuse.lam, w0))));
                  const float n1 = __fsub_rn(w1, __fmul_rn(p.fuse.eM, __fadd_rn(__fmul_rn(fd->shape_scale, bf_hi(xw[e])),
                                                                               __fmul_rn(p.fuse.lam, w1))));
                  ww[e] = pack_bf2(n0, n1);
                }
                *reinterpret_cast<uint4*>(wcol + (int64_t)ii * fd->cols) = make_uint4(ww[0], ww[1], ww[2], ww[3]);
              }
            }
          }
        }
      } else if (kP == 1 && lane == 0 && warp_in && !split) {
        // the boxes went out from the chunk loop (boxes past the padded
        // columns hold nothing and were skipped there); auxbuf may be
        // rewritten once the stores have read it
        bulk_wait_read();
      }
      __syncwarp();
      if (aux_phase) {
        if (lane == 0) mbar_arrive(aux_empty);
        xph ^= 1u;
      }
    }
    if (lane == 0) bulk_wait_all();
  }

  __syncwarp();
  pair_finish<kStages>(*log, abort_flag, full, R.armed, rank);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// Split Gram tiles: bf16 A tile = the sum of the fp32 parts (already scaled),
// added in part order.
__global__ void __launch_bounds__(256) ns_split_finish_kernel(const NsSplitTarget* __restrict__ targets,
                                                              const float* __restrict__ ws, const unsigned* flags) {
  asm volatile("griddepcontrol.wait;" ::: "memory");   // the Gram launch before it may be programmatic
  if (lm_stopped(flags)) return;
  const NsSplitTarget T = targets[blockIdx.y];
  __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(T.a_tile);
  // four consecutive elements of a row per thread and trip (the tile's
  // column extent is a multiple of 128): 16-byte loads of every part, 8-byte
  // stores per plane; each element's parts are still added in part order
  for (int e = (blockIdx.x * blockDim.x + threadIdx.x) * 4; e < BM * BN; e += gridDim.x * blockDim.x * 4) {
    const int r = e / BN, c = e % BN;
    if (r >= T.nr || c >= T.nc) continue;
    float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
    const float* part = ws + (size_t)T.first * (BM * BN) + e;
#pragma unroll 4
    for (int k = 0; k < T.nparts; ++k) {
      const float4 v = __ldg(reinterpret_cast<const float4*>(part + (size_t)k * (BM * BN)));
      sum.x += v.x;
      sum.y += v.y;
      sum.z += v.z;
      sum.w += v.w;
    }
    const size_t o = (size_t)r * T.ld + c;
    if (T.plane == 0) {
      *reinterpret_cast<uint2*>(dst + o) = make_uint2(pack_bf2(sum.x, sum.y), pack_bf2(sum.z, sum.w));
    } else {   // three bf16 planes
      float h[4], m[4], l[4];
      split3(sum.x, h[0], m[0], l[0]);
      split3(sum.y, h[1], m[1], l[1]);
      split3(sum.z, h[2], m[2], l[2]);
      split3(sum.w, h[3], m[3], l[3]);
      *reinterpret_cast<uint2*>(dst + o) = make_uint2(pack_bf2(h[0], h[1]), pack_bf2(h[2], h[3]));
      *reinterpret_cast<uint2*>(dst + T.plane + o) = make_uint2(pack_bf2(m[0], m[1]), pack_bf2(m[2], m[3]));
      *reinterpret_cast<uint2*>(dst + 2 * T.plane + o) = make_uint2(pack_bf2(l[0], l[1]), pack_bf2(l[2], l[3]));
    }
  }
}

// Diagnostic: one thread waits, with the same bounded wait as the NS kernel,
// on an mbarrier nobody arrives on; when the limit passes it records
// LM_FLAG_TIMEOUT and returns normally.
__global__ void bounded_wait_probe_kernel(uint64_t limit_ns, unsigned* flags) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    if (!mbar_wait(&bar, 0, &abort_flag, limit_ns)) atomicOr(flags, LM_FLAG_TIMEOUT);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  }
  return fn;
}

cudaError_t encode_3d(CUtensorMap* m, void* base, uint64_t inner, uint64_t rows, uint64_t count,
                      uint32_t box_inner, uint32_t box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
  if (enc == nullptr) return cudaErrorNotSupported;
  const cuuint64_t dims[3] = {inner, rows, count};
  const cuuint64_t strides[2] = {inner * 2, inner * rows * 2};
  const cuuint32_t box[3] = {box_inner, box_rows, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// MN-major operand map: dimensions (64, rows, inner / 64, count), the third
// 128 bytes apart, box (64, box_k, 2, 1): one copy reads a 128-wide half.
cudaError_t encode_mn4d(CUtensorMap* m, void* base, uint64_t inner, uint64_t rows, uint64_t count,
                        uint32_t box_k) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
  if (enc == nullptr) return cudaErrorNotSupported;
  const cuuint64_t dims[4] = {64, rows, inner / 64, count};
  const cuuint64_t strides[3] = {inner * 2, 128, inner * rows * 2};
  const cuuint32_t box[4] = {64, box_k, 2, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, base, dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_bounded_wait_probe(uint64_t limit_ns, unsigned* flags, cudaStream_t st) {
  count_launch();
  bounded_wait_probe_kernel<<<1, 32, 0, st>>>(limit_ns, flags);
  return cudaGetLastError();
}

cudaError_t tc_encode_w_maps(void* w, int64_t rows, int64_t cols, CUtensorMap* maps) {
  // W (rows x cols bf16, row-major, cols % 8 = 0, 16-byte aligned) as a 3-D
  // tensor of one matrix: loads of 64 x 128 boxes, stores of 64 x 32 boxes
  if (rows <= 0 || cols <= 0 || (cols & 7) != 0 || (reinterpret_cast<uintptr_t>(w) & 15) != 0)
    return cudaErrorInvalidValue;
  cudaError_t e = encode_3d(&maps[0], w, (uint64_t)cols, (uint64_t)rows, 1, BK, kHalf);
  if (e == cudaSuccess) e = encode_3d(&maps[1], w, (uint64_t)cols, (uint64_t)rows, 1, 64, 32);
  return e;
}

int tc_pad_s(int s) { return (s + kHalf - 1) / kHalf * kHalf; }
int tc_pad_l(int l) { return (l + BN - 1) / BN * BN; }

cudaError_t tc_encode_group_maps(const NsGroup& g, TcGroupMaps* maps, int pieces) {
  cudaError_t e;
  // three-piece buffers hold piece q of matrix k as matrix k + q * count
  const uint64_t nm = (uint64_t)g.count * (uint64_t)pieces;
  // X buffers: s_pad x l_pad (wide) or l_pad x s_pad (tall), row-major
  const uint64_t inner = g.tall ? g.s_pad : g.l_pad, rows = g.tall ? g.l_pad : g.s_pad;
  for (int b = 0; b < 2; ++b) {
    if ((e = encode_3d(&maps->xk[b], g.X[b], inner, rows, nm, BK, kHalf)) != cudaSuccess) return e;
    if ((e = encode_3d(&maps->xst[b], g.X[b], inner, rows, nm, 64, 32)) != cudaSuccess) return e;
    if ((e = encode_mn4d(&maps->xmn[b], g.X[b], inner, rows, nm, BK)) != cudaSuccess) return e;
  }
  if ((e = encode_3d(&maps->a, g.A, g.s_pad, g.s_pad, nm, BK, kHalf)) != cudaSuccess) return e;
  if ((e = encode_3d(&maps->b, g.B, g.s_pad, g.s_pad, nm, BK, kHalf)) != cudaSuccess) return e;
  if ((e = encode_mn4d(&maps->amn, g.A, g.s_pad, g.s_pad, nm, BK)) != cudaSuccess) return e;
  if ((e = encode_mn4d(&maps->bmn, g.B, g.s_pad, g.s_pad, nm, BK)) != cudaSuccess) return e;
  if ((e = encode_3d(&maps->ast, g.A, g.s_pad, g.s_pad, nm, 64, 32)) != cudaSuccess) return e;
  if ((e = encode_3d(&maps->bst, g.B, g.s_pad, g.s_pad, nm, 64, 32)) != cudaSuccess) return e;
  return cudaSuccess;
}

namespace {
__global__ void __launch_bounds__(256) split3_kernel(const float4* __restrict__ src, uint2* __restrict__ dst,
                                                     size_t n4, const unsigned* flags) {
  if (lm_stopped(flags)) return;
  for (size_t k = blockIdx.x * (size_t)blockDim.x + threadIdx.x; k < n4; k += (size_t)gridDim.x * blockDim.x) {
    const float4 v = src[k];
    float h[4], m[4], l[4];
    split3(v.x, h[0], m[0], l[0]);
    split3(v.y, h[1], m[1], l[1]);
    split3(v.z, h[2], m[2], l[2]);
    split3(v.w, h[3], m[3], l[3]);
    dst[k] = make_uint2(pack_bf2(h[0], h[1]), pack_bf2(h[2], h[3]));
    dst[n4 + k] = make_uint2(pack_bf2(m[0], m[1]), pack_bf2(m[2], m[3]));
    dst[2 * n4 + k] = make_uint2(pack_bf2(l[0], l[1]), pack_bf2(l[2], l[3]));
  }
}
}  // namespace

cudaError_t launch_split3(const float* src, void* dst, size_t n, const unsigned* flags, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  if (n % 4 != 0) return cudaErrorInvalidValue;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const size_t n4 = n / 4;
  size_t grid = (n4 + 255) / 256;
  if (grid > (size_t)sms * 8) grid = (size_t)sms * 8;
  count_launch();
  split3_kernel<<<(unsigned)grid, 256, 0, st>>>(reinterpret_cast<const float4*>(src), static_cast<uint2*>(dst), n4, flags);
  return cudaGetLastError();
}

cudaError_t launch_ns_split_finish(const NsSplitTarget* targets, int n, const float* ws, const unsigned* flags,
                                   cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  count_launch();
  ns_split_finish_kernel<<<dim3(32, n), 256, 0, st>>>(targets, ws, flags);
  return cudaGetLastError();
}

int tc_max_pairs() {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return sms / 2 > 0 ? sms / 2 : 1;
}

template <bool kMasked, bool kSplit, int kP>
static cudaError_t set_smem_attr() {
  return cudaFuncSetAttribute(ns_tc_kernel<kMasked, kSplit, kP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)TcLayout<kP>::kSmemBytes);
}

cudaError_t launch_ns_tc(NsPhase ph, int iter, int ngroups, const NsGroup* groups,
                         const TcGroupMaps* maps, const NsTile* tiles, int ntiles,
                         const int* offsets, int npairs, const double* norm2, NsCoeffs co,
                         unsigned* flags, const FuseFinal* fuse, cudaStream_t st,
                         const unsigned char* active, float* split_ws, int pieces, int final_f32, bool wide,
                         bool pdl, uint64_t wait_ns, bool apply_from_a, bool fold_a) {
  if (ntiles <= 0) return cudaSuccess;
  if (apply_from_a && (ph != NS_APPLY || wide)) return cudaErrorInvalidValue;
  if (fold_a && (ph == NS_GRAM || wide || pieces != 1 || apply_from_a)) return cudaErrorInvalidValue;
  if (ngroups < 1 || ngroups > kMaxGroupsTc) return cudaErrorInvalidValue;
  if (pieces != 1 && pieces != 3) return cudaErrorInvalidValue;
  if (pieces == 3 && (fuse != nullptr || wide)) return cudaErrorInvalidValue;
  if (wait_ns == 0) return cudaErrorInvalidValue;
  static bool attr_set[kMaxDevices] = {};
  const int slot = device_slot();
  if (slot < 0 || !attr_set[slot]) {
    cudaError_t e = set_smem_attr<false, false, 1>();
    if (e == cudaSuccess) e = set_smem_attr<true, false, 1>();
    if (e == cudaSuccess) e = set_smem_attr<false, true, 1>();
    if (e == cudaSuccess) e = set_smem_attr<true, true, 1>();
    if (e == cudaSuccess) e = set_smem_attr<false, false, 3>();
    if (e == cudaSuccess) e = set_smem_attr<true, false, 3>();
    if (e == cudaSuccess) e = set_smem_attr<false, true, 3>();
    if (e == cudaSuccess) e = set_smem_attr<true, true, 3>();
    if (e != cudaSuccess) return e;
    if (slot >= 0) attr_set[slot] = true;
  }
  TcParams prm;
  memset(&prm, 0, sizeof(prm));
  for (int gi = 0; gi < ngroups; ++gi) {
    prm.maps[gi] = maps[gi];
    prm.groups[gi] = groups[gi];
  }
  prm.tiles = tiles;
  prm.offsets = offsets;
  prm.ntiles = ntiles;
  prm.phase = (int)ph;
  prm.iter = iter;
  prm.norm2 = norm2;
  prm.co = co;
  prm.apply_from_a = apply_from_a ? 1 : 0;
  prm.fold_a = fold_a ? 1 : 0;
  prm.flags = flags;
  if (fuse != nullptr && ph == NS_APPLY) prm.fuse = *fuse;
  prm.active = active;
  prm.split_ws = split_ws;
  prm.final_f32 = (pieces == 3 && ph == NS_APPLY && final_f32) ? 1 : 0;
  prm.wait_ns = wait_ns;
  int pairs = npairs;
  if (offsets == nullptr) {
    pairs = tc_max_pairs();
    if (pairs > ntiles) pairs = ntiles;
  }
  const int grid = 2 * (pairs > 0 ? pairs : 1);
  const bool split = split_ws != nullptr && ph == NS_GRAM;
  const bool masked = active != nullptr;
  if (wide) return launch_ns_wide(prm, grid, masked, split, pdl, st);
  count_launch();
  if (pieces == 3) {
    constexpr size_t sm = TcLayout<3>::kSmemBytes;
    if (masked) {
      if (split) return launch_tc_kernel(ns_tc_kernel<true, true, 3>, grid, sm, pdl, st, prm);
      return launch_tc_kernel(ns_tc_kernel<true, false, 3>, grid, sm, pdl, st, prm);
    }
    if (split) return launch_tc_kernel(ns_tc_kernel<false, true, 3>, grid, sm, pdl, st, prm);
    return launch_tc_kernel(ns_tc_kernel<false, false, 3>, grid, sm, pdl, st, prm);
  }
  constexpr size_t sm = TcLayout<1>::kSmemBytes;
  if (masked) {
    if (split) return launch_tc_kernel(ns_tc_kernel<true, true, 1>, grid, sm, pdl, st, prm);
    return launch_tc_kernel(ns_tc_kernel<true, false, 1>, grid, sm, pdl, st, prm);
  }
  if (split) return launch_tc_kernel(ns_tc_kernel<false, true, 1>, grid, sm, pdl, st, prm);
  return launch_tc_kernel(ns_tc_kernel<false, false, 1>, grid, sm, pdl, st, prm);
}

}  // namespace lm
