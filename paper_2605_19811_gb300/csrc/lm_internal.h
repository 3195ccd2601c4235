// Internal declarations shared by the library's translation units: device
// tables built by lm_create and the launchers each kernel file provides.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "lionmuon.h"

namespace lm {

constexpr int kPtrsPerUpload = 1024;   // pointers per pointer-upload launch

#ifdef __CUDACC__
// Every kernel of a step reads the status word at entry: once a bounded wait
// has given up (LM_FLAG_TIMEOUT), the rest of the step, and every later
// step until the flag is cleared, does nothing.  NULL: no status word.
__device__ __forceinline__ bool lm_stopped(const unsigned* flags) {
  return flags != nullptr && (*reinterpret_cast<const volatile unsigned*>(flags) & LM_FLAG_TIMEOUT) != 0u;
}
#endif

// ---------------------------------------------------------------------------
// Lion multi-tensor step (Algorithm 1, Lion branch + momentum update)
// ---------------------------------------------------------------------------
struct LionTensor {
  void* w;         // bf16 or fp32 parameter (dtype fixed per table)
  float* m;        // fp32 momentum
  int64_t n;       // elements
  int32_t grad_slot;   // index into the device grad-pointer table
  int32_t pad;
};
struct LionChunk {
  int32_t tensor;  // index into the LionTensor table
  int32_t pad;
  int64_t begin;   // first element (multiple of 8)
  int64_t count;   // elements
};
struct LionConsts {
  float b1, c1, b2, c2, eL, lam;
  // Adaptive selection: skip[param] != 0 makes the Lion kernel leave that
  // parameter alone (it takes the Muon step); NULL: no parameter skipped.
  const unsigned char* skip;
  const unsigned* flags;   // status word read at entry (lm_stopped), or NULL
};

// AdamW on 1-D parameters (the LM_VECTOR_ADAMW rule): parameter, first
// moment (the momentum buffer), second moment, chunked like the Lion tables.
struct AdamTensor {
  void* w;
  float* m;
  float* v;
  int64_t n;
  int32_t grad_slot;
  int32_t pad;
};
// float32 constants of one step: b1, 1-b1, b2, 1-b2, lr/(1-b1^k),
// 1/sqrt(1-b2^k), lr*wd, eps (k = t + 1), each rounded once from double.
struct AdamConsts {
  float b1, c1, b2, c2, step, rbc2, lrwd, eps;
  const unsigned* flags;   // status word read at entry (lm_stopped), or NULL
};
cudaError_t launch_adamw(lm_dtype dt, const AdamTensor* tensors, const LionChunk* chunks, int nchunks,
                         const void* const* grads, AdamConsts k, cudaStream_t st);

// Launch the Lion kernel over a chunk table whose tensors all have dtype dt.
cudaError_t launch_lion(lm_dtype dt, const LionTensor* tensors, const LionChunk* chunks,
                        int nchunks, const void* const* grads, LionConsts k,
                        int grid, cudaStream_t st);
int lion_grid_size(lm_dtype dt);
// Momentum update alone over a chunk table (matrices another rank owns on a
// layer-sharded Muon step); k.b2, k.c2 and k.flags are used.
cudaError_t launch_ema(lm_dtype dt, const LionTensor* tensors, const LionChunk* chunks, int nchunks,
                       const void* const* grads, LionConsts k, int grid, cudaStream_t st);

// ---------------------------------------------------------------------------
// Muon element-wise kernels: momentum + norm -> X0 (K2), finalize (K6)
// ---------------------------------------------------------------------------
struct MatDesc {
  void* w;          // parameter (rows x cols, dtype wdt); for msign: the input
  float* m;         // momentum (NULL for msign: no momentum)
  void* x;          // X buffer base for this matrix (the parameter's orientation, padded)
  void* x_final;    // the buffer holding X_K after the NS iterations
  void* out;        // msign output (rows x cols, dtype odt), or NULL
  double* norm2;    // Frobenius-norm^2 accumulator of G_hat
  int64_t rows, cols;
  int64_t ldx;      // row pitch of X (elements): l_pad (wide) or s_pad (tall)
  int32_t grad_slot;
  int32_t pad_;
  int32_t wdt;      // lm_dtype of w (and the gradient)
  int32_t odt;      // lm_dtype of out
  float shape_scale;    // 0.2*sqrt(max(rows, cols))
};
// A range of elements of one matrix (row-major over rows x cols); begin is a
// multiple of 8.
struct ElemChunk {
  int32_t mat;
  int32_t pad_;
  int64_t begin;
  int64_t count;
};
constexpr int64_t kElemChunk = 32768;   // elements per chunk
struct MuonConsts {
  float b1, c1, b2, c2;   // interpolation / momentum constants
  float eM, lam;          // Muon learning rate and weight decay
  float eps;              // NS normalisation eps
  int32_t ns_steps;
  // Adaptive selection: active[mat] != 0 for the matrices that take the
  // Muon step; NULL: every matrix does.
  const unsigned char* active;
  const unsigned* flags;   // status word read at entry (lm_stopped), or NULL
};
// mode 0: Muon momentum step (G_hat from grads + momentum, M update)
// mode 1: msign input (G_hat = input tensor, no momentum)
// gdt: dtype of every chunk's gradient (mode 0) or input (mode 1).
cudaError_t launch_momentum_norm(lm_dtype xdt, lm_dtype gdt, const MatDesc* mats, const ElemChunk* chunks,
                                 int nchunks, const void* const* grads, MuonConsts k,
                                 int mode, cudaStream_t st);
// mode 0: W <- W - eM (scale X_K' + lam W); mode 1: out = X_K'
// where X_K' = X_K, or X_K / (||G_hat|| + eps) when ns_steps == 0.
// pdt: dtype of every chunk's parameter (mode 0) or output (mode 1).
cudaError_t launch_finalize(lm_dtype xdt, lm_dtype pdt, const MatDesc* mats, const ElemChunk* chunks,
                            int nchunks, MuonConsts k, int mode, unsigned* flags,
                            cudaStream_t st);

// ---------------------------------------------------------------------------
// Newton-Schulz GEMM phases (grouped over same-shape matrices)
// ---------------------------------------------------------------------------
enum NsPhase { NS_GRAM = 0, NS_POLY = 1, NS_APPLY = 2 };

struct NsGroup {
  int32_t count;          // matrices in the group
  int32_t s, l;           // true sizes (s = min, l = max)
  int32_t s_pad, l_pad;   // padded sizes of the workspace buffers
  int32_t first_mat;      // index of the group's first matrix in the norm array
  int32_t tall;           // 1: X kept as l x s (rows > cols), 0: as s x l
  int32_t pad_;
  void* X[2];             // ping-pong X: count x (s_pad x l_pad, or l_pad x s_pad if tall)
  void* A;                // count x s_pad x s_pad
  void* B;                // count x s_pad x s_pad
  // Three-piece tensor-core mode: X, A and B hold three bf16 planes (piece q
  // of matrix k is matrix k + q * count of the buffer), and Xf is an fp32
  // count x s_pad x l_pad buffer for X_0 (from the momentum kernel) and X_K.
  void* Xf;
};
// Tile work item: group, matrix-in-group, tile row, tile col.
struct NsTile {
  uint16_t group, mat, tm, tn;
  // Split-K (Gram phase only): K blocks [kb0, kb1) of the tile, kb1 == 0 for
  // all of them; slot != 0: the partial product is written in fp32 to
  // workspace tile slot - 1 instead of A (NsSplitTarget sums the parts).
  uint16_t kb0, kb1, slot;
  // 256-column output blocks of the tile, starting at block tn: 2 only in
  // the wide-tile kernel's launches (0 and 1 both mean one block).
  uint16_t nh;
};
// A split Gram tile (tile edge `tile`: 256 tensor-core, 128 fp32 path): the
// parts in workspace tiles first .. first + nparts - 1 are summed in that
// order (so the result does not depend on timing) and written to A at
// (tm * tile + r, tn * tile + c) for r < nr, c < nc; the fp32 path, which keeps
// A whole, also writes the mirror (tn * tile + c, tm * tile + r), and on a
// diagonal tile only c >= r.
struct NsSplitTarget {
  void* a_tile;           // element (tm * tile, tn * tile) of the matrix's A
  void* a_mirror;         // element (tn * tile, tm * tile) (fp32 path)
  int32_t ld;             // s_pad
  int32_t nr, nc;         // rows / columns of the tile inside the padded matrix
  int32_t first, nparts;
  int32_t diag;
  int64_t plane;          // three-piece A: elements between its bf16 planes (0: one bf16 plane)
};
constexpr int kMaxGroupsTc = 8;   // groups per tensor-core launch

struct NsCoeffs {
  float a, b, c, eps;
};

// Tensor-core path (bf16 operands, fp32 accumulation in TMEM): one
// kTcBM x kTcBN output tile per CTA pair; s is padded to 128, l to kTcBN.
constexpr int kTcBM = 256, kTcBN = 256, kTcBK = 64;
int tc_pad_s(int s);
int tc_pad_l(int l);
// Tensor maps for one group: K-major boxes (64 x 128), MN-major boxes
// (64 x 64) and store boxes (64 x 32) on X0, X1, A, B.  A and B hold only
// their 256 x 256 tiles on or above the diagonal.
struct TcGroupMaps {
  CUtensorMap xk[2];    // K-major operand / aux loads: box 64 x 128
  CUtensorMap a;
  CUtensorMap b;
  CUtensorMap xmn[2];   // MN-major operand loads: 4-D box (64, 64, 2), a 128-wide half
  CUtensorMap amn;      // transposed reads of stored A / B tiles: the same 4-D box
  CUtensorMap bmn;
  CUtensorMap xst[2];   // result stores: box 64 x 32
  CUtensorMap ast;
  CUtensorMap bst;
};
// pieces: 1 (bf16 buffers) or 3 (three bf16 planes per buffer)
cudaError_t tc_encode_group_maps(const NsGroup& g, TcGroupMaps* maps, int pieces = 1);
int tc_max_pairs();   // CTA pairs that fit the device (one CTA per SM)
// One bounded wait on a barrier that is never signalled (failure-detection probe).
cudaError_t launch_bounded_wait_probe(uint64_t limit_ns, unsigned* flags, cudaStream_t st);
// The Muon parameter write fused into the epilogue of the last APPLY phase:
// W <- W - eM (shape_scale X_K + lam W) for the bf16 parameters of mats
// (indexed by group first_mat + matrix), X_K itself is not stored.
struct FuseFinal {
  const MatDesc* mats;
  float eM, lam;
  // Two TMA maps per matrix (same index as mats), in device memory: W as
  // 64 x 128 load boxes and 64 x 32 store boxes (tc_encode_w_maps).  Used
  // where a is folded into B' (the APPLY then has no X tile to read).
  const CUtensorMap* wmaps;
};
// The two W maps of FuseFinal::wmaps for one bf16 parameter (cols % 8 = 0).
cudaError_t tc_encode_w_maps(void* w, int64_t rows, int64_t cols, CUtensorMap* maps);
// Limit of a bounded device wait unless the state sets another
// (LM_WAIT_LIMIT_NS at lm_create): a wait that runs out gives up and raises
// LM_FLAG_TIMEOUT; every later kernel then does nothing until the flag is cleared.
constexpr uint64_t kDefaultWaitNs = 5000000000ull;   // 5 s
uint64_t env_wait_limit_ns();   // LM_WAIT_LIMIT_NS if set to a positive integer, else kDefaultWaitNs
// offsets: NULL (round robin over tiles) or npairs + 1 range starts;
// fuse: NULL, or the parameter write of the last APPLY phase;
// apply_from_a: an APPLY of an iteration whose c is 0, whose POLY launch was
// left out (B = b A): it reads A and scales its product by b (one-block
// tiles only).
cudaError_t launch_ns_tc(NsPhase ph, int iter, int ngroups, const NsGroup* groups,
                         const TcGroupMaps* maps, const NsTile* tiles, int ntiles,
                         const int* offsets, int npairs, const double* norm2, NsCoeffs co,
                         unsigned* flags, const FuseFinal* fuse, cudaStream_t st,
                         const unsigned char* active = nullptr, float* split_ws = nullptr, int pieces = 1,
                         int final_f32 = 0, bool wide = false, bool pdl = false,
                         uint64_t wait_ns = kDefaultWaitNs, bool apply_from_a = false, bool fold_a = false);
// split_ws: non-NULL only for a Gram launch whose tiles include split-K parts.
// pieces = 3: fp32 operands as three bf16 pieces (no split tiles, no fused
// parameter write); final_f32: this APPLY writes fp32 X to NsGroup::Xf.
// wide: the tile list may hold two-block tiles (NsTile::nh = 2), run by the
// wide-tile kernel (bf16 only); pdl: programmatic dependent launch (the
// kernel may start while the previous kernel on the stream finishes).
// Both kernels do nothing when LM_FLAG_TIMEOUT is already set in *flags.
// fp32 -> three bf16 planes (hi, mid, lo; their sum is exactly the input):
// n elements of src, plane q at dst + q * n.
cudaError_t launch_split3(const float* src, void* dst, size_t n, const unsigned* flags, cudaStream_t st);
// After a Gram launch with split tiles: bf16 A tiles from the fp32 parts.
cudaError_t launch_ns_split_finish(const NsSplitTarget* targets, int n, const float* ws, const unsigned* flags,
                                   cudaStream_t st);

// fp32 CUDA-core path.
constexpr int kSimtBM = 128, kSimtBN = 128;
int simt_pad(int x);
cudaError_t launch_ns_simt(NsPhase ph, int iter, int ngroups, const NsGroup* dgroups,
                           const NsTile* tiles, int ntiles, const double* norm2, NsCoeffs co,
                           cudaStream_t st, const unsigned char* active = nullptr, float* split_ws = nullptr,
                           const unsigned* flags = nullptr);
// fp32 path: A tiles (and mirrors) from the fp32 parts of split Gram tiles.
cudaError_t launch_ns_split_finish_f32(const NsSplitTarget* targets, int n, const float* ws, const unsigned* flags,
                                       cudaStream_t st);
// active (both NS paths): NULL, or active[first_mat + mat] != 0 for the
// matrices whose tiles run; tiles of the others are skipped by every role.

// Power iteration for the stable-rank selection (Appendix G).  One pass
// reads each matrix M (fp32 momentum, row-major) once: with v the input
// vector normalised, u = M v row by row, ||u||^2 into acc[1 + pass], and
// (unless last) M^T u added into the output vector; pass 0 also adds
// ||M||_F^2 into acc[0].  Pass k reads v0 (k = 0), wa (k odd) or wb (k even)
// and writes wa (k even) or wb (k odd), which must be zero beforehand.
struct SrMat {
  const float* M;
  const float* v0;
  float* wa;
  float* wb;
  double* acc;            // 1 + passes doubles, zero before pass 0
  int64_t rows, cols;
  int32_t mat, param;     // matrix id (NS numbering) and parameter index
};
constexpr int kSrankRows = 64;   // rows per power-iteration work item
struct SrItem {
  int32_t m;              // index into the SrMat table
  int32_t row0, nrows;    // rows of this work item
  int32_t pad;
};
// Launch shape for a column count: slots per thread and threads per block;
// slots = 0 means cols is too large (more than 16384).
int srank_slots(int64_t cols, int* threads);
cudaError_t launch_srank_pass(int slots, int threads, bool vec4, const SrMat* mats, const SrItem* items,
                              int nitems, int pass, bool last, const unsigned* flags, cudaStream_t st);
// The same pass through the shared-memory ring (every matrix of the launch
// with cols % 4 == 0, at most max_cols <= 16384 columns); a stalled copy sets
// LM_FLAG_TIMEOUT in *flags.
// Launch shape of the ring kernel for rows of `cols` columns as one code
// (100 x consumer warps + slots per thread; 0 beyond 16384 columns): rows
// with the same code share a launch.
int srank_ring_shape(int64_t cols);
cudaError_t launch_srank_ring(int max_cols, const SrMat* mats, const SrItem* items, int nitems, int pass, bool last,
                              unsigned* flags, uint64_t wait_ns, cudaStream_t st);
// Decide per matrix: Muon iff ||M||_F^2 == 0 or ||M||_F^2 <= alpha min(m, n)
// sigma^2 (sigma^2 = acc[1 + last_pass]); writes active[mat], skip[param]
// and the estimate srank[mat] = ||M||_F^2 / sigma^2.
cudaError_t launch_srank_decide(const SrMat* mats, int nmat, double alpha, int last_pass, unsigned char* active,
                                unsigned char* skip, double* srank, const unsigned* flags, cudaStream_t st);
constexpr int kMaxGroupsSimt = 64;

// Launch accounting (lm_kernel_launch_count) and the thread's last-error text.
void count_launch();
// Per-device slot for the launchers' one-time set-ups (kernel attributes set
// and grid sizes read on each device the process uses): the current device,
// or -1 when it cannot be used as an index (beyond kMaxDevices).
constexpr int kMaxDevices = 64;
int device_slot();
lm_status set_error(lm_status st, const char* msg);

// Pointer table upload (grads) as a kernel with the pointers in its parameters.
struct PtrUpload {
  const void* p[kPtrsPerUpload];
};
cudaError_t launch_upload_ptrs(const void** dst, const PtrUpload& src, int count,
                               cudaStream_t st);

}  // namespace lm
