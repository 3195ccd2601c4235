// Definitions shared by the two tensor-core Newton-Schulz kernels:
//   lm_ns_tc.cu   one 256 x 256 output tile per CTA pair, two accumulators
//                 in TMEM (bf16 operands, or fp32 as three bf16 pieces);
//   lm_ns_wide.cu tiles of one or two 256-column halves per CTA pair (bf16),
//                 which reuse one staged A box for both halves.
// Both run the NS phases of Section 2's iteration (GRAM A = X X^T, POLY
// B = b A + c A A, APPLY X' = a X + B X) on CTA pairs (cta_group::2) with
// operands staged by TMA, and share the launch parameters, the start-of-launch
// stop check and the end-of-launch handshake that makes a give-up safe.
#pragma once

#include "lm_internal.h"
#include "lm_tc_ptx.cuh"

namespace lm {

constexpr int kNsThreads = 32 * 11;   // producer, MMA/TMEM, 8 epilogue warps, aux loader

struct TcParams {
  TcGroupMaps maps[kMaxGroupsTc];
  NsGroup groups[kMaxGroupsTc];
  const NsTile* tiles;
  const int* offsets;   // tiles of pair k: [offsets[k], offsets[k+1]); NULL: round robin
  int ntiles;
  int phase;
  int iter;
  const double* norm2;
  NsCoeffs co;
  unsigned* flags;
  FuseFinal fuse;       // fuse.mats != NULL: this APPLY writes the parameters
  const unsigned char* active;   // NULL, or per matrix: 0 = skip its tiles
  float* split_ws;               // fp32 workspace of split Gram tiles (256 x 256 each)
  int final_f32;                 // three-piece operands: this APPLY writes fp32 X to NsGroup::Xf
  uint64_t wait_ns;              // limit of every bounded wait of the roles
  int apply_from_a;              // APPLY of an iteration with c = 0: B = b A was not formed,
                                 // the left operand is A and the accumulator is scaled by b
  int fold_a;                    // POLY adds a to B's diagonal (B' = a I + B); APPLY is X' = B' X
};

// Launch of the wide-tile kernel (lm_ns_wide.cu); grid = 2 x CTA pairs.
cudaError_t launch_ns_wide(const TcParams& prm, int grid, bool masked, bool split, bool pdl, cudaStream_t st);
// cudaLaunchKernelEx with the programmatic-stream-serialisation attribute
// (when pdl): the launch may begin before the previous kernel on the stream
// ends, and its kernel waits (griddepcontrol.wait) before touching anything
// that kernel wrote.
template <typename Kern>
cudaError_t launch_tc_kernel(Kern kernel, int grid, size_t smem, bool pdl, cudaStream_t st, const TcParams& prm) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid, 1, 1);
  cfg.blockDim = dim3(kNsThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, prm);
}

namespace tcs {
namespace {

constexpr int BM = kTcBM, BN = kTcBN, BK = kTcBK;   // 256 x 256 output blocks, K step 64
constexpr int kHalf = 128;                           // A rows / B N-rows per CTA
constexpr int kABytes = kHalf * BK * 2;              // 16 KB
constexpr int kBBytes = kHalf * BK * 2;              // 16 KB
static_assert(kABytes == kBBytes, "diagonal tiles read their A boxes as B");
constexpr int kEpiWarps = 8;
constexpr int kAuxWarp = 2 + kEpiWarps;              // warp that loads the epilogue's aux boxes
constexpr int kThreads = kNsThreads;
static_assert(kThreads == 32 * (3 + kEpiWarps), "role layout");
constexpr int kAuxBoxBytes = kHalf * 64 * 2;         // one 64-column box of the CTA's rows: 16 KB
constexpr uint64_t kCleanupWaitNs = 100000000ull;    // waits for in-flight copies after a give-up

// Whether a tile's matrix runs in this launch; every role asks the same
// question of the same tiles, so skipping keeps their pipelines in step.
__device__ __forceinline__ bool tile_active(const TcParams& p, const NsTile& t) {
  return p.active == nullptr || p.active[p.groups[t.group].first_mat + t.mat] != 0;
}

// Start of a launch, after the barriers and TMEM are set up (every thread of
// both CTAs).  Waits for the kernel this launch depends on, then returns
// whether the launch must do nothing because an earlier kernel gave up a
// bounded wait (LM_FLAG_TIMEOUT).  CTA 0 of the pair reads the status word
// and CTA 1 takes CTA 0's answer, so both CTAs agree even if another pair
// of this launch raises the flag meanwhile.
__device__ __forceinline__ bool pair_start(const TcParams& p, uint32_t* stop_word, uint32_t rank) {
  tc::griddep_wait();
  if (threadIdx.x == 0)
    *stop_word = rank == 0 ? ((*reinterpret_cast<volatile unsigned*>(p.flags) & LM_FLAG_TIMEOUT) != 0u) : 0u;
  tc::tc_fence_before();
  tc::cluster_sync();   // barriers of both CTAs initialised, CTA 0's answer visible
  tc::tc_fence_after();
  const bool stop = tc::ld_peer_u32(stop_word, 0) != 0u;
  tc::griddep_launch_dependents();
  return stop;
}

// What each CTA's producer records for the end-of-launch handshake, and the
// copy of the peer CTA's record that the peer writes into this CTA.
template <int kStages>
struct ProducerLog {
  uint32_t n;                  // K blocks whose copies this CTA issued
  uint32_t bytes[kStages];     // bytes this CTA copied for the last K block of each stage
  uint32_t peer_n, peer_abort, peer_bytes[kStages];   // written by the peer CTA
};

// End of a launch (every thread of both CTAs, after all roles have left
// their loops; thread 0 is the producer lane).  Both CTAs' copies of a K
// block signal CTA 0's full barrier, which CTA 0's producer arms with both
// CTAs' bytes; the MMA issuer waits for all its MMAs before it gets here.
// When every role finished normally both producers issued the same K blocks
// and everything they copied has been consumed.  After a give-up (any role of
// either CTA) one producer may have issued K blocks the other did not: CTA 0
// then arms the barrier for CTA 1's copies that it never armed, or lowers the
// expected count by the share CTA 1 never copied, waits (bounded) until every
// armed stage has landed, and only then do the CTAs pass a second cluster
// barrier and leave.  No copy is in flight into a CTA, or signalling a barrier
// of a CTA, that has exited.  Each CTA writes its record into the peer before
// the first cluster barrier, so nothing reads a peer's shared memory after a
// barrier the peer may already have left by.  armed[s]: parity of the last
// phase CTA 0 armed on stage s, or -1 (CTA 0's producer lane only).
template <int kStages>
__device__ __forceinline__ void pair_finish(ProducerLog<kStages>& log, const volatile int* abort_flag, uint64_t* full,
                                            int* armed, uint32_t rank) {
  __syncwarp();
  __syncthreads();   // every role of this CTA is done: the log and the abort word are final
  const uint32_t peer = rank ^ 1u;
  if (threadIdx.x == 0) {
    tc::st_peer_u32(&log.peer_n, peer, log.n);
    tc::st_peer_u32(&log.peer_abort, peer, *abort_flag != 0 ? 1u : 0u);
    for (int s = 0; s < kStages; ++s) tc::st_peer_u32(&log.peer_bytes[s], peer, log.bytes[s]);
  }
  tc::tc_fence_before();
  tc::cluster_sync();   // A: both records are in both CTAs
  const bool ab = *abort_flag != 0 || log.peer_abort != 0u;
  if (!ab && log.n == log.peer_n) return;   // same decision in both CTAs: the inputs are symmetric
  if (rank == 0 && threadIdx.x == 0) {
    const uint32_t n0 = log.n, n1 = log.peer_n;
    for (uint32_t j = min(n0, n1); j < max(n0, n1); ++j) {
      const int s = (int)(j % (uint32_t)kStages);
      if (n1 > n0) {
        // CTA 1 copied K block j, CTA 0 never armed it
        tc::mbar_arrive_expect_tx(&full[s], log.peer_bytes[s]);
        armed[s] = (int)((j / (uint32_t)kStages) & 1u);
      } else {
        // CTA 0 armed K block j for both CTAs, CTA 1 never copied its share
        // (the same boxes of its own rows, so the same byte count)
        tc::mbar_complete_tx(&full[s], log.bytes[s]);
      }
    }
    volatile int never = 0;
    for (int s = 0; s < kStages; ++s)
      if (armed[s] >= 0) tc::mbar_wait(&full[s], (uint32_t)armed[s], &never, kCleanupWaitNs);
  }
  __syncwarp();
  tc::cluster_sync();   // B: nothing is in flight into either CTA any more
}

}  // namespace
}  // namespace tcs
}  // namespace lm
