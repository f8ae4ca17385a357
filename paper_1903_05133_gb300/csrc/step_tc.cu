// bf16 learner step on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
// One local SGD step of Algorithm 1 (Sec. 3.1) for every learner of a ReLU MLP:
// forward Z_l = H_{l-1} W_l^T + b_l, softmax cross-entropy gradient, backward
// dH_{l-1} = dZ_l W_l (with W_l before its update) and W_l -= lr * dZ_l^T H_{l-1}.
// The fp32 master weights W_l [P][out][in] are streamed from HBM by TMA and
// rounded to bf16 by the CTA itself into tensor memory; MMAs accumulate in fp32 in
// tensor memory.  Activations exist once, batch-major ([Bn][features], 128-byte
// swizzled tiles): the forward reads them K-major, the backward's dW MMA MN-major.
//
// Because the per-learner batch B (<= 64) is far below the MMA's M, every GEMM
// is issued "swap-AB": the weight tile supplies M = 128 rows and the batch is
// the N extent.  Both kernels are persistent stream-K kernels (one CTA per SM):
//   forward:  unit = 128 output features x 64 inputs of one learner;
//             Z^T[128 x Bn] += W_q H^T, epilogue bias + ReLU (or fused softmax-CE);
//   backward: unit = 128 input features x 64 output rows of one learner;
//             dW^T = H^T dZ, the fp32 update of W, and dH^T += W_q^T dZ^T;
//             epilogue dZ_{l-1} = dH [H_{l-1} > 0], b_{l-1} -= lr sum_b dZ_{l-1}.
// W is read once by the forward and once (read, written) by the backward.
#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "ptx.cuh"

namespace ha {
namespace {


// ------------------------------------------------------------------ forward
// Forward of one layer on the tensor cores.  The work is a list of tiles: tile =
// (learner j, 128 output features), reduced over the layer's input in chunks of 64
// features.  Two schedules:
//  * Dynamic (layers with many tiles).  Work items are handed out from a global
//    counter, so an SM that streams its weights faster simply takes more of them
//    (per-SM streaming rates differ by up to 1.8x under full load, and a static split
//    waits for the slowest SM).  Most tiles are one item each.  The tiles of the
//    last clusters of learners (the "tail": at least one tile per SM) are split into
//    fixed pieces of kPieceChunks chunks, so that the work left at the end is fine
//    grained.  Which tiles are split and where depends on the layer's shape only.
//    Each piece writes its partial sum to a slot of its own; the piece that
//    completes a tile (an atomic count per tile) adds the tile's partials in piece
//    order and runs the epilogue.  The sum of every output therefore has one fixed
//    order, whichever CTA computed which piece.  No CTA waits for another.
//  * Cluster split-K (layers with at most 76 tiles): tile t gets a cluster of cq
//    CTAs, rank k taking chunks [k*nk/cq, (k+1)*nk/cq); at the end ranks 1.. leave
//    their partial in shared memory and rank 0 adds them in rank order through
//    distributed shared memory and runs the epilogue.
// Warps 0-7 convert the fp32 weight tiles to bf16 and own the accumulator rows:
// warp w serves TMEM lanes 32*(w%4).., converts K half w/4 of those 32 rows, and
// the two warps on the same lanes split the batch columns in interleaved 16-column
// blocks (group w/4 takes blocks 2m + w/4).  Warp 8 claims the work items and
// streams the weight tiles, warp 9 issues the MMAs, warp 10 streams the batch tiles.
// Every role that waits has a warp of its own: a lane blocked in an mbarrier wait
// would hold up the other lanes of its warp.  Warp 8 announces each claimed item to
// the other roles through a small queue in shared memory.
// The bf16 A tile (128 rows x 64 K) lives in tensor memory, double-buffered, so
// shared memory holds only the two TMA rings: the fp32 weight tiles (two
// 128-byte-swizzled 128 x 32 boxes per chunk, released by the converter warps as
// soon as they have read them, so conversion and MMA latency stay out of the
// weight stream) and the bf16 batch tiles (Bn x 128 bytes, released by the MMA),
// plus (fused cross-entropy only) a staging area for the epilogue.  A chunk takes
// about 4-5 us from TMA issue to arrival under full load, so both rings are as deep
// as shared memory allows.
// Right after a compact local average the learners of a cluster read their cluster's
// mean (TcFwdArgs::w_div > 1); k_tc_forward_group then forwards groups of them at once.
constexpr int kFwdConv = 256;
constexpr int kFwdThreads = kFwdConv + 96;
constexpr int kFwdWRingMax = 6, kFwdHRingMax = 8;
constexpr int kFwdWf32 = 128 * 64 * 4;                 // 32 KB fp32 W tile (2 boxes)
constexpr int kFwdWBox = 128 * 32 * 4;                 // one 128 x 32 fp32 box
constexpr int kFwdSmemMax = 227 * 1024;
constexpr int kXentSmem = (2 * 128 * 65 + 4 * 64) * 4; // logits, gradients, statistics
constexpr int kBarBytes = 768;                         // mbarriers, queue, flags
// The tensor core's fp32 accumulation loses precision roughly in proportion to the
// number of MMAs chained into one accumulator, so the accumulator is promoted:
// every kSegChunks chunks (16 MMAs) the partial sum is folded into fp32 registers
// with IEEE adds, in chunk order, while the MMAs continue in the other TMEM buffer.
constexpr int kSegChunks = 4;
// TMEM columns: accumulators at 0 and 64, bf16 A tiles (32 columns each) at 128, 160.
constexpr uint32_t kFwdTmemCols = 256;
constexpr uint32_t kFwdTmemA = 128;
constexpr int kFwdHidden = 0, kFwdXent = 2;   // TcFwdArgs::mode (1 = logits)
constexpr int kQueue = 8;                     // claimed work items announced ahead

// Layout: W ring | epilogue staging (mode 2) | batch ring | barriers.
__host__ __device__ constexpr int fwd_wring(int mode, int Bn) {
  return mode == 2 ? 3 : (Bn <= 32 ? 6 : 5);
}
__host__ __device__ constexpr int fwd_h_off(int mode, int Bn) {
  return fwd_wring(mode, Bn) * kFwdWf32 + (mode == 2 ? kXentSmem : 0);
}
__host__ __device__ constexpr int fwd_hring(int mode, int Bn) {
  return (kFwdSmemMax - 1024 - kBarBytes - fwd_h_off(mode, Bn)) / (Bn * 128) < kFwdHRingMax
             ? (kFwdSmemMax - 1024 - kBarBytes - fwd_h_off(mode, Bn)) / (Bn * 128)
             : kFwdHRingMax;
}
__host__ __device__ constexpr int fwd_bar_off(int mode, int Bn) {
  return fwd_h_off(mode, Bn) + fwd_hring(mode, Bn) * Bn * 128;
}
__host__ __device__ constexpr int fwd_smem(int mode, int Bn) {
  return fwd_bar_off(mode, Bn) + kBarBytes + 1024;
}
static_assert(fwd_hring(2, 64) >= 6 && fwd_hring(0, 64) == 8 && fwd_hring(0, 32) == 8 &&
                  fwd_smem(2, 64) <= kFwdSmemMax && fwd_smem(0, 64) <= kFwdSmemMax &&
                  fwd_smem(0, 48) <= kFwdSmemMax && fwd_smem(0, 32) <= kFwdSmemMax &&
                  fwd_smem(0, 16) <= kFwdSmemMax && fwd_smem(2, 16) <= kFwdSmemMax,
              "forward shared-memory plan");

// Bounded wait whose outcome is made uniform across the warp, so that a warp never
// reaches a .sync.aligned tcgen05 instruction with only some of its lanes.
__device__ __forceinline__ bool wait_warp(uint64_t* bar, uint32_t parity, int* err) {
  const bool r = mbar_wait(bar, parity, err);
  return __all_sync(0xffffffffu, r);
}

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(p);
  return reinterpret_cast<uint8_t*>((a + 1023) & ~uintptr_t(1023));
}

// A barrier of the converter threads on an mbarrier, bounded like every other
// wait.  `phase` counts this thread's uses.
struct GroupSync {
  uint64_t* bar;
  uint32_t phase;
  int* err;
  __device__ __forceinline__ bool operator()() {
    mbar_arrive(bar);
    const bool ok = mbar_wait(bar, phase & 1, err);
    ++phase;
    return ok;
  }
};

// One work item of a forward layer: chunks [c_lo, c_hi) of tile tau (learner
// tau / o_tiles, outputs 128 * (tau % o_tiles) ..), piece `piece` of the tile's np
// pieces (np = 1: the whole tile).
struct FwdItem {
  int tau, c_lo, c_hi, piece, np;
};

// Tiles per learner and the row divisor of the weights a kernel reads (> 1: the
// learners of a cluster read the same row of the cluster means).
__device__ __forceinline__ int item_span(const TcFwdArgs& a) { return a.o_tiles; }
__device__ __forceinline__ int item_span(const TcBwdArgs& a) { return a.s_tiles; }
__device__ __forceinline__ int item_div(const TcFwdArgs& a) { return a.w_div; }
__device__ __forceinline__ int item_div(const TcBwdArgs& a) { return a.src_div; }

// Work item `it` of the dynamic schedule: items [0, n_whole) are the whole tiles
// [0, n_whole); then come the pieces of the tail tiles [n_whole, n_tiles), tile by
// tile, the pieces of a tile in order.  Whole tiles go in tile order, except when the
// learners of a cluster share their weights (item_div > 1): within each cluster whose
// tiles are all whole, its learners' tiles with the same weight tile are claimed one
// after the other, so that they stream the same weight rows at about the same time and
// L2 serves all but the first.  (The split into whole and tail tiles is unchanged, so
// every tile is summed the same way.)
template <class Args>
__device__ __forceinline__ FwdItem fwd_item(const Args& a, int nk, int it) {
  FwdItem f;
  if (it < a.n_whole) {
    f.tau = it;
    const int S = item_div(a);
    if (S > 1) {
      const int span = item_span(a), blk = S * span, c = it / blk;
      if ((c + 1) * blk <= a.n_whole) {
        const int r = it - c * blk, o = r / S, m = r - o * S;
        f.tau = c * blk + m * span + o;
      }
    }
    f.c_lo = 0;
    f.c_hi = nk;
    f.piece = 0;
    f.np = 1;
  } else {
    const int np = a.np_tail, i2 = it - a.n_whole, tt = i2 / np, p = i2 - tt * np;
    f.tau = a.n_whole + tt;
    f.c_lo = p * a.piece_chunks;
    f.c_hi = f.c_lo + a.piece_chunks < nk ? f.c_lo + a.piece_chunks : nk;
    f.piece = p;
    f.np = np;
  }
  return f;
}

// The update+forward kernel's order (uf_item): that of fwd_item, extended to the
// clusters whose tiles are partly tail and to the tail.  After an average its first
// step reads the weights from the cluster means; so that the learners of a cluster
// claim the same weight rows together there too, the whole tiles of a partly-tail
// cluster go over its whole learners (when they end on a learner boundary), and the
// tail, when made of whole learners, goes over them piece by piece (tail tile m * span
// + o, piece p, in the order (o, p, m)).  DRAM reads of that launch with 8 learners of
// 12288-4096-4096-1000, where half the tiles are tail: 0.45 instead of 0.95 GB.  (The
// same order in the forward and the backward measured no faster, the backward slower.)
__device__ __forceinline__ FwdItem uf_item(const TcFwdArgs& a, int nk, int it) {
  FwdItem f;
  const int S = a.w_div, span = a.o_tiles;
  if (it < a.n_whole) {
    f.tau = it;
    if (S > 1) {
      const int blk = S * span, base = it / blk * blk, rem = a.n_whole - base;
      const int mc = rem >= blk ? S : (rem % span == 0 ? rem / span : 0);
      if (mc > 1) {
        const int r = it - base, o = r / mc, m = r - o * mc;
        f.tau = base + m * span + o;
      }
    }
    f.c_lo = 0;
    f.c_hi = nk;
    f.piece = 0;
    f.np = 1;
  } else {
    const int np = a.np_tail, i2 = it - a.n_whole, t_tail = a.n_tiles - a.n_whole;
    int tt = i2 / np, p = i2 - tt * np;
    if (S > 1 && t_tail % span == 0 && t_tail > span) {
      const int mt = t_tail / span, rest = i2 / mt, m = i2 - rest * mt, o = rest / np;
      p = rest - o * np;
      tt = m * span + o;
    }
    f.tau = a.n_whole + tt;
    f.c_lo = p * a.piece_chunks;
    f.c_hi = f.c_lo + a.piece_chunks < nk ? f.c_lo + a.piece_chunks : nk;
    f.piece = p;
    f.np = np;
  }
  return f;
}

// The queue through which the claiming warp announces work items: items[q] holds
// the k-th claimed item (k % kQueue == q), -1 once there are no more.
struct ItemQueue {
  uint64_t* full;    // [kQueue] item written
  uint64_t* empty;   // [kQueue] read by every consuming warp
  int* items;        // [kQueue]
  // Producer (one lane): publish the k-th item.
  __device__ __forceinline__ bool put(int k, int it, int* err) {
    const int q = k % kQueue;
    if (k >= kQueue && !mbar_wait(&empty[q], ((k / kQueue) - 1) & 1, err)) return false;
    items[q] = it;
    mbar_arrive(&full[q]);
    return true;
  }
  // Consumer (a whole warp): the k-th item, read by every lane; lane 0 then frees the
  // slot for this warp.  -1: no more items (or a wait expired).
  __device__ __forceinline__ int take(int k, int lane, int* err) {
    const int q = k % kQueue;
    if (!wait_warp(&full[q], (k / kQueue) & 1, err)) return -1;
    const int it = items[q];
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[q]);
    return it;
  }
};

// The partial of a split tile: written by its piece, read by the piece that
// completes the tile.  Slot (tail tile tt, piece p) = part[((tt * np + p) * 128 + r) * Bn].
__device__ __forceinline__ void store_partial(float* dst, const float* acc, int gr, int Bn) {
#pragma unroll
  for (int m = 0; m < 2; ++m) {
    const int cb = (2 * m + gr) * 16;
    if (cb < Bn) {
#pragma unroll
      for (int q = 0; q < 16; q += 4)
        __stcg(reinterpret_cast<float4*>(dst + cb + q),
               make_float4(acc[16 * m + q], acc[16 * m + q + 1], acc[16 * m + q + 2],
                           acc[16 * m + q + 3]));
    }
  }
}

// A piece of a split tile ends: its partial goes to its slot; the piece that
// completes the tile (the last to count itself in) replaces acc with the sum of all
// the tile's partials in piece order (P_0 + P_1 + ... with IEEE fp32 adds, its own
// read back like the others) and returns true: it runs the epilogue.  Every
// converter thread calls it (`flag` is a shared word; false on an expired wait too).
__device__ __forceinline__ bool piece_end(const TcFwdArgs& a, const FwdItem& f, int t, int r, int gr,
                                          float* acc, GroupSync& gsync, volatile int* flag,
                                          bool& ok) {
  const int tt = f.tau - a.n_whole;
  const float* slots = a.part + static_cast<int64_t>(tt) * f.np * 128 * a.Bn;
  store_partial(a.part + ((static_cast<int64_t>(tt) * f.np + f.piece) * 128 + r) * a.Bn, acc, gr,
                a.Bn);
  if (!gsync()) { ok = false; return false; }   // every converter thread's partial is written
  if (t == 0) {
    fence_acq_rel_gpu();           // release: the CTA's partial before the count
    const int before = atomicAdd(a.counters + tt, 1);
    const int last = before == f.np - 1;
    if (last) {
      fence_acq_rel_gpu();         // acquire: every other piece's partial before the reads
      a.counters[tt] = 0;          // ready for the next launch
    }
    *flag = last;
  }
  if (!gsync()) { ok = false; return false; }
  if (!*flag) return false;
  // acc = P_0 + P_1 + ... in piece order; the loads of two pieces are in flight at once
  for (int m = 0; m < 2; ++m) {
    const int cb = (2 * m + gr) * 16;
    if (cb >= a.Bn) continue;
#pragma unroll
    for (int q = 0; q < 16; q += 4) {
      const float* src = slots + static_cast<int64_t>(r) * a.Bn + cb + q;
      const int64_t pstride = static_cast<int64_t>(128) * a.Bn;
      float4 s0 = __ldcg(reinterpret_cast<const float4*>(src));
      for (int p = 1; p < f.np; p += 2) {
        const float4 v1 = __ldcg(reinterpret_cast<const float4*>(src + p * pstride));
        float4 v2 = make_float4(0.f, 0.f, 0.f, 0.f);
        if (p + 1 < f.np) v2 = __ldcg(reinterpret_cast<const float4*>(src + (p + 1) * pstride));
        s0.x = __fadd_rn(s0.x, v1.x);
        s0.y = __fadd_rn(s0.y, v1.y);
        s0.z = __fadd_rn(s0.z, v1.z);
        s0.w = __fadd_rn(s0.w, v1.w);
        if (p + 1 < f.np) {
          s0.x = __fadd_rn(s0.x, v2.x);
          s0.y = __fadd_rn(s0.y, v2.y);
          s0.z = __fadd_rn(s0.z, v2.z);
          s0.w = __fadd_rn(s0.w, v2.w);
        }
      }
      acc[16 * m + q] = s0.x;
      acc[16 * m + q + 1] = s0.y;
      acc[16 * m + q + 2] = s0.z;
      acc[16 * m + q + 3] = s0.w;
    }
  }
  return true;
}

// Epilogue of the last layer when every class fits in one 128-row tile: the
// softmax cross-entropy gradient straight from the accumulator (no logits
// round trip).  Row r = class, group gr holds the column blocks 2m + gr of it
// (blocks of 16 samples) in acc[16m ..].  Work is then spread over all converter
// threads: column statistics, all class x sample gradients, per-class bias sums
// in sample order.
__device__ __forceinline__ void xent_epilogue(const TcFwdArgs& a, int j, int t, int r, int gr,
                                              const float* acc, float* sm, GroupSync& gsync) {
  constexpr int ZP = 65;
  float* zs = sm;                  // [128][ZP] logits, class-major
  float* gs = sm + 128 * ZP;       // [128][ZP] gradients
  float* stat = gs + 128 * ZP;     // max[64], sum[64], label[64], loss[64]
  const int C = a.out, B = a.B;
  if (r < C) {
#pragma unroll
    for (int m = 0; m < 2; ++m) {
      const int cb = (2 * m + gr) * 16;
      if (cb < a.Bn) {
#pragma unroll
        for (int q = 0; q < 16; ++q) zs[r * ZP + cb + q] = acc[16 * m + q];
      }
    }
  }
  gsync();
  if (t < B) {
    float m = -INFINITY;
    for (int c = 0; c < C; ++c) m = fmaxf(m, zs[c * ZP + t]);
    float s = 0.f;
    for (int c = 0; c < C; ++c) s += expf(zs[c * ZP + t] - m);
    const int yb = a.y[static_cast<int64_t>(j) * a.N + (a.row0 + t) % a.N];
    stat[t] = m;
    stat[64 + t] = s;
    stat[128 + t] = __int_as_float(yb);
    stat[192 + t] = logf(s) + m - zs[yb * ZP + t];
  }
  gsync();
  const float fB = static_cast<float>(B);
  for (int e = t; e < C * B; e += kFwdConv) {
    const int c = e / B, b = e - c * B;
    const float p = __fdiv_rn(expf(zs[c * ZP + b] - stat[b]), stat[64 + b]);
    const float g = __fdiv_rn(__fsub_rn(p, __float_as_int(stat[128 + b]) == c ? 1.f : 0.f), fB);
    gs[c * ZP + b] = g;
    a.dz_out[(static_cast<int64_t>(j) * a.Bn + b) * a.pitch_out + c] = __float2bfloat16_rn(g);
  }
  gsync();
  if (t == 0) {
    float l = 0.f;
    for (int b = 0; b < B; ++b) l += stat[192 + b];
    a.loss[j] = l / B;
  }
  if (t < C) {
    float db = 0.f;
    for (int b = 0; b < B; ++b) db = __fadd_rn(db, gs[t * ZP + b]);
    const float bv = a.bias[static_cast<int64_t>(j / a.b_div) * a.ld + t];
    a.bias_out[static_cast<int64_t>(j) * a.ld + t] = __fsub_rn(bv, __fmul_rn(a.lr, db));
  }
  gsync();   // the staging area is reused by the next tile
}

// kDyn: dynamic work items (compiled separately from cluster split-K, so that each
// schedule carries only its own code and registers).
template <bool kDyn>
__global__ void __launch_bounds__(kFwdThreads, 1)
    k_tc_forward(const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_h,
                 const TcFwdArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = blockIdx.x;
  const int nk = (a.in + 63) / 64;
  constexpr bool dyn = kDyn;
  const int cq = kDyn ? 1 : a.cq, part = g % cq;           // cluster split-K rank
  const int n_items = a.n_whole + (a.n_tiles - a.n_whole) * a.np_tail;
  const int nw = fwd_wring(a.mode, a.Bn), nh = fwd_hring(a.mode, a.Bn);
  const int hbytes = a.Bn * 128;
  const int h_row0 = a.x_direct ? a.x_row0 : 0;           // batch rows inside the H (or X) map
  uint8_t* xent_sm = smem + nw * kFwdWf32;
  uint8_t* h_base = smem + fwd_h_off(a.mode, a.Bn);
  uint64_t* wfull = reinterpret_cast<uint64_t*>(smem + fwd_bar_off(a.mode, a.Bn));
  uint64_t* wempty = wfull + kFwdWRingMax;  // weight tile read by every converter warp
  uint64_t* hfull = wempty + kFwdWRingMax;
  uint64_t* hempty = hfull + kFwdHRingMax;  // batch tile consumed by the MMA
  uint64_t* conv = hempty + kFwdHRingMax;   // [2] A tile written to TMEM
  uint64_t* wfree = conv + 2;              // [2] A tile consumed by the MMA
  uint64_t* accf = wfree + 2;              // [2] accumulator segment complete
  uint64_t* accr = accf + 2;               // [2] accumulator segment drained
  uint64_t* gbar = accr + 2;               // converter-group barrier
  uint64_t* done = gbar + 1;
  ItemQueue queue{done + 1, done + 1 + kQueue, nullptr};
  queue.items = reinterpret_cast<int*>(done + 1 + 2 * kQueue);
  int* last_flag = queue.items + kQueue;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(last_flag + 1);
  auto wf = [&](int s) { return smem + s * kFwdWf32; };
  auto hb = [&](int s) { return h_base + s * hbytes; };
  // Cluster split-K: this CTA's one item.  Dynamic: the k-th claimed item.
  const FwdItem cl_item{g / cq, part * nk / cq, (part + 1) * nk / cq, 0, 1};
  constexpr int kConsumers = 2 + kFwdConv / 32;            // MMA, batch and converter warps

  if (threadIdx.x == 0) {
    for (int s = 0; s < kFwdWRingMax; ++s) {
      mbar_init(&wfull[s], 1);
      mbar_init(&wempty[s], kFwdConv / 32);   // one arrival per converter warp
    }
    for (int s = 0; s < kFwdHRingMax; ++s) {
      mbar_init(&hfull[s], 1);
      mbar_init(&hempty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&conv[b], kFwdConv / 32);
      mbar_init(&wfree[b], 1);
      mbar_init(&accf[b], 1);
      mbar_init(&accr[b], kFwdConv);
    }
    if (dyn)
      for (int q = 0; q < kQueue; ++q) {
        mbar_init(&queue.full[q], 1);
        mbar_init(&queue.empty[q], kConsumers);
      }
    mbar_init(gbar, kFwdConv);
    mbar_init(done, 1);
    fence_barrier_init();
  }
  if (warp == 9) {
    tmem_alloc(tmem_slot, kFwdTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  grid_dep_wait();                       // the previous kernel's results are visible

  // The k-th item of this CTA for a consuming warp (-1: none left).
  auto next_item = [&](int k, FwdItem& f) -> bool {
    if (!dyn) {
      f = cl_item;
      return k == 0;
    }
    const int it = queue.take(k, lane, a.err);
    if (it < 0) return false;
    f = fwd_item(a, nk, it);
    return true;
  };

  if (warp == 8) {
    if (lane == 0) {
      // claim (dynamic), announce, and stream the weight tiles (kept in L2 as usual when
      // the learners of a cluster read the same ones)
      tma_prefetch_desc(&tm_w);
      const uint64_t stream = l2_weight_policy(a.w_stream != 0, a.w_div > 1);
      int i = 0, issued = 0;
      bool ok = true;
      int next = dyn ? atomicAdd(a.dyn, 1) : 0;
      for (int k = 0; ok; ++k) {
        FwdItem f;
        if (dyn) {
          const int it = next < n_items ? next : -1;
          if (!queue.put(k, it, a.err) || it < 0) break;
          next = atomicAdd(a.dyn, 1);           // the next claim, hidden behind these loads
          f = fwd_item(a, nk, it);
        } else {
          if (k > 0) break;
          f = cl_item;
        }
        const int j = f.tau / a.o_tiles, ot = f.tau - j * a.o_tiles;
        // learner j's weights: row j / w_div of the map (the cluster means right after a
        // compact local average)
        const int jw = j / a.w_div;
        for (int c = f.c_lo; c < f.c_hi; ++c, ++i) {
          const int s = i % nw;
          if (i >= nw && !mbar_wait(&wempty[s], ((i / nw) - 1) & 1, a.err)) { ok = false; break; }
          mbar_arrive_expect_tx(&wfull[s], kFwdWf32);
          tma_load_3d_hint(wf(s), &tm_w, &wfull[s], c * 64, ot * 128, jw, stream);
          tma_load_3d_hint(wf(s) + kFwdWBox, &tm_w, &wfull[s], c * 64 + 32, ot * 128, jw, stream);
          issued = i + 1;
        }
      }
      // Every load issued must have landed before the CTA may exit.
      for (int u = issued - nw > 0 ? issued - nw : 0; u < issued; ++u)
        mbar_wait(&wfull[u % nw], (u / nw) & 1, a.err);
    }
    if (cq > 1) {
      cluster_sync_all();   // the two barriers of the cluster reduction (see below)
      cluster_sync_all();
    }
  } else if (warp == 10) {
    // batch tiles
    if (lane == 0) tma_prefetch_desc(&tm_h);
    int i = 0, issued = 0;
    bool ok = true;
    FwdItem f;
    for (int k = 0; ok && next_item(k, f); ++k) {
      if (lane == 0) {
        const int j = f.tau / a.o_tiles;
        for (int c = f.c_lo; c < f.c_hi; ++c, ++i) {
          const int s = i % nh;
          if (i >= nh && !mbar_wait(&hempty[s], ((i / nh) - 1) & 1, a.err)) { ok = false; break; }
          mbar_arrive_expect_tx(&hfull[s], a.Bn * 128);
          tma_load_3d(hb(s), &tm_h, &hfull[s], c * 64, h_row0, j);
          issued = i + 1;
        }
      }
      ok = __all_sync(0xffffffffu, ok);
    }
    if (lane == 0)
      for (int u = issued - nh > 0 ? issued - nh : 0; u < issued; ++u)
        mbar_wait(&hfull[u % nh], (u / nh) & 1, a.err);
    if (cq > 1) {
      cluster_sync_all();
      cluster_sync_all();
    }
  } else if (warp == 9) {
    const uint32_t idesc = umma_idesc_bf16(128, a.Bn);
    int q = -1, i = 0;                 // accumulator segment index, chunk counter
    bool ok = true;
    FwdItem f;
    for (int k = 0; ok && next_item(k, f); ++k) {
      if (lane == 0) {
        for (int c = f.c_lo, p = 0; c < f.c_hi; ++c, ++p, ++i) {
          const bool tlast = c == f.c_hi - 1;
          const bool first = p % kSegChunks == 0, last = tlast || p % kSegChunks == kSegChunks - 1;
          const int sh = i % nh, b = i & 1;
          if (first) ++q;
          const int ab = q & 1;
          if (first && q >= 2 && !mbar_wait(&accr[ab], ((q >> 1) - 1) & 1, a.err)) { ok = false; break; }
          if (!mbar_wait(&conv[b], (i >> 1) & 1, a.err)) { ok = false; break; }
          if (!mbar_wait(&hfull[sh], (i / nh) & 1, a.err)) { ok = false; break; }
          tc_fence_after();
          const uint32_t at = tmem + kFwdTmemA + 32 * b;
          const uint64_t bd = umma_desc_sw128(smem_u32(hb(sh)));
          const uint32_t d = tmem + 64 * ab;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_bf16_ta(d, at + 8 * kk, bd + 2 * kk, idesc, (!first || kk > 0) ? 1u : 0u);
          tc_commit(&hempty[sh]);
          tc_commit(&wfree[b]);
          if (last) tc_commit(&accf[ab]);
        }
      }
      ok = __all_sync(0xffffffffu, ok);
    }
    if (lane == 0) {
      tc_commit(done);
      mbar_wait(done, 0, a.err);   // no MMA may be in flight at teardown
    }
    if (cq > 1) {
      cluster_sync_all();
      cluster_sync_all();
    }
  } else {
    // ---- warps 0-7: fp32 -> bf16 A tile, the accumulator drains and the epilogues
    const int t = threadIdx.x;
    const int r = t & 127, gr = t >> 7;                    // accumulator row, column group
    const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
    GroupSync gsync{gbar, 0, a.err};
    float acc[32];                                         // blocks 2m + gr, m = 0, 1
#pragma unroll
    for (int q = 0; q < 32; ++q) acc[q] = 0.f;
    int qc = -1, drained = 0;
    // Fold segment `drained` into the registers (warp-uniform; contains tcgen05.ld).
    auto drain = [&]() -> bool {
      const int ab = drained & 1;
      if (!wait_warp(&accf[ab], (drained >> 1) & 1, a.err)) return false;
      tc_fence_after();
#pragma unroll
      for (int m = 0; m < 2; ++m) {
        const int cb = (2 * m + gr) * 16;
        if (cb < a.Bn) {
          float v[16];
          tmem_ld16(tbase + 64 * ab + cb, v);
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 16; ++q) acc[16 * m + q] = __fadd_rn(acc[16 * m + q], v[q]);
        }
      }
      tc_fence_before();
      mbar_arrive(&accr[ab]);
      ++drained;
      return true;
    };
    // Tile tau's sum is in acc: bias, activation or cross-entropy, store.
    auto epilogue = [&](int tau, float bias) {
      const int j = tau / a.o_tiles, ot = tau - j * a.o_tiles;
      const int o = ot * 128 + r;
      const bool valid = o < a.out;
      if (a.mode == kFwdXent) {
#pragma unroll
        for (int q = 0; q < 32; ++q) acc[q] = __fadd_rn(acc[q], bias);
        xent_epilogue(a, j, t, r, gr, acc, reinterpret_cast<float*>(xent_sm), gsync);
      } else if (valid) {
#pragma unroll
        for (int m = 0; m < 2; ++m) {
          const int cb = (2 * m + gr) * 16;
          if (cb >= a.Bn) break;
          if (a.mode == kFwdHidden) {
#pragma unroll
            for (int q = 0; q < 16; ++q)
              if (cb + q < a.B)
                a.h_out[(static_cast<int64_t>(j) * a.Bn + cb + q) * a.pitch_out + o] =
                    __float2bfloat16_rn(fmaxf(__fadd_rn(acc[16 * m + q], bias), 0.f));
          } else {
#pragma unroll
            for (int q = 0; q < 16; ++q)
              if (cb + q < a.B)
                a.z_out[(static_cast<int64_t>(j) * a.B + cb + q) * a.out + o] = __fadd_rn(acc[16 * m + q], bias);
          }
        }
      }
    };
    bool ok = true;
    int i = 0;
    int ep_tau = -1;                   // cluster split-K: this CTA's tile
    float ep_bias = 0.f;
    FwdItem f;
    for (int k = 0; ok && next_item(k, f); ++k) {
      const int j = f.tau / a.o_tiles, ot = f.tau - j * a.o_tiles;
      const int ob = ot * 128 + r;
      const float tbias = ob < a.out ? a.bias[static_cast<int64_t>(j / a.b_div) * a.ld + ob] : 0.f;
      for (int c = f.c_lo, p = 0; c < f.c_hi && ok; ++c, ++p, ++i) {
        const bool tlast = c == f.c_hi - 1;
        const int sw = i % nw, bb = i & 1;
        if (!wait_warp(&wfull[sw], (i / nw) & 1, a.err)) { ok = false; break; }
        if (i >= 2 && !wait_warp(&wfree[bb], ((i >> 1) - 1) & 1, a.err)) { ok = false; break; }
        tc_fence_after();
        {
          // Row 32*(warp%4) + lane, K half warp/4: 32 floats from the swizzled box
          // (16-byte chunk q of row r sits at chunk q ^ (r%8)), packed to bf16 pairs,
          // stored as 16 TMEM columns of this lane.
          const int row = 32 * (warp & 3) + lane, half = warp >> 2;
          const uint8_t* src = wf(sw) + half * kFwdWBox + row * 128;
          uint32_t pk[16];
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            const float4 x = *reinterpret_cast<const float4*>(src + ((q ^ (row & 7)) << 4));
            pk[2 * q] = pack_bf16x2(x.x, x.y);
            pk[2 * q + 1] = pack_bf16x2(x.z, x.w);
          }
          tmem_st16(tbase + kFwdTmemA + 32 * bb + 16 * half, pk);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&wempty[sw]);   // the fp32 tile is no longer needed
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&conv[bb]);
        if (p % kSegChunks == 0) ++qc;
        if (tlast) {
          while (ok && drained <= qc)
            if (!drain()) ok = false;
          if (!ok) break;
          if (!dyn) {
            // cluster split-K: rank 0 keeps its partial in registers, the others
            // leave theirs in the (now idle) weight ring for rank 0 to read
            ep_tau = f.tau;
            ep_bias = tbias;
            if (part != 0) {
              float* red = reinterpret_cast<float*>(smem) + r * a.Bn;
#pragma unroll
              for (int m = 0; m < 2; ++m) {
                const int cb = (2 * m + gr) * 16;
                if (cb < a.Bn) {
#pragma unroll
                  for (int q = 0; q < 16; q += 4)
                    *reinterpret_cast<float4*>(red + cb + q) =
                        make_float4(acc[16 * m + q], acc[16 * m + q + 1], acc[16 * m + q + 2],
                                    acc[16 * m + q + 3]);
                }
              }
            }
          } else {
            const bool fin = f.np == 1 || piece_end(a, f, t, r, gr, acc, gsync, last_flag, ok);
            if (ok && fin) epilogue(f.tau, tbias);
#pragma unroll
            for (int q = 0; q < 32; ++q) acc[q] = 0.f;
            ok = __all_sync(0xffffffffu, ok);
          }
        } else if (p % kSegChunks == kSegChunks - 1 && qc >= 1 && drained < qc) {
          if (!drain()) ok = false;   // one segment behind the MMAs
        }
      }
    }
    if (cq > 1) {
      // Cluster split-K finish: rank 0 adds the partials of ranks 1.. (left in their
      // shared memory) in rank order and runs the epilogue.  (Splitting the epilogue
      // by column blocks across the ranks measured slower.)
      cluster_sync_all();   // the partials of ranks 1.. are in their shared memory
      if (part == 0 && __all_sync(0xffffffffu, ok && ep_tau >= 0)) {
        for (int rk = 1; rk < cq; ++rk) {
          const float* red = reinterpret_cast<const float*>(smem) + r * a.Bn;
#pragma unroll
          for (int m = 0; m < 2; ++m) {
            const int cb = (2 * m + gr) * 16;
            if (cb < a.Bn) {
#pragma unroll
              for (int q = 0; q < 16; q += 4) {
                const float4 v = ld_cluster_f4(red + cb + q, rk);
                acc[16 * m + q] = __fadd_rn(acc[16 * m + q], v.x);
                acc[16 * m + q + 1] = __fadd_rn(acc[16 * m + q + 1], v.y);
                acc[16 * m + q + 2] = __fadd_rn(acc[16 * m + q + 2], v.z);
                acc[16 * m + q + 3] = __fadd_rn(acc[16 * m + q + 3], v.w);
              }
            }
          }
        }
        epilogue(ep_tau, ep_bias);
      }
      cluster_sync_all();   // rank 0 has read them: every CTA may exit
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kFwdTmemCols);
  }
  if (dyn && threadIdx.x == 0) {
    // the last CTA out resets the claim counters for the next launch (every claim of
    // every CTA precedes that CTA's increment here)
    __threadfence();
    if (atomicAdd(a.dyn + 1, 1) == static_cast<int>(gridDim.x) - 1) {
      a.dyn[0] = 0;
      a.dyn[1] = 0;
    }
  }
}


// ------------------------------------------------------------------ grouped forward
// Right after a compact local average the learners of a cluster hold the same weights,
// their cluster's mean.  The forward of G learners of a cluster is then one product of
// each weight tile of the mean with their G stacked batch tiles (N = G * Bn <= 128
// columns): a weight chunk is streamed and converted once for G learners instead of G
// times.  Every output (learner, sample) is summed exactly as k_tc_forward sums it: the
// same chunks, the same every-kSegChunks promotion from the item's first chunk, the
// same pieces added in piece order, and the columns of one MMA do not mix, so the bits
// are the per-learner forward's.  Work item = group tile (learners q*G .. q*G+G-1,
// outputs 128*ot ..): whole group tiles first, then the pieces of the tail group tiles;
// the plan's tail must consist of whole groups (n_whole a multiple of G * o_tiles).
// Hidden layers (mode 0) and logits (mode 1).  Roles as in k_tc_forward.
constexpr int kGfWRing = 5;
constexpr uint32_t kGfTmemCols = 512;          // accumulators at 0 and 128, A tiles at 256
constexpr uint32_t kGfTmemA = 256;
// A tiles in flight (32 TMEM columns each): the converters run up to kGfABufs chunks
// ahead of the MMA, which covers their pause at every accumulator drain.
constexpr int kGfABufs = 4;
static_assert(kGfTmemA + 32 * kGfABufs <= kGfTmemCols && (kGfABufs & (kGfABufs - 1)) == 0,
              "grouped forward TMEM plan");
__host__ __device__ constexpr int gf_h_off() { return kGfWRing * kFwdWf32; }
__host__ __device__ constexpr int gf_hring(int N) {
  return (kFwdSmemMax - 1024 - kBarBytes - gf_h_off()) / (N * 128) < kFwdHRingMax
             ? (kFwdSmemMax - 1024 - kBarBytes - gf_h_off()) / (N * 128)
             : kFwdHRingMax;
}
__host__ __device__ constexpr int gf_bar_off(int N) { return gf_h_off() + gf_hring(N) * N * 128; }
__host__ __device__ constexpr int gf_smem(int N) { return gf_bar_off(N) + kBarBytes + 1024; }
static_assert(gf_hring(128) >= 4 && gf_smem(128) <= kFwdSmemMax && gf_smem(96) <= kFwdSmemMax,
              "grouped forward shared-memory plan");

struct GfItem {
  int q, ot, c_lo, c_hi, piece, np;
};

// Group tiles in claim order q-major.  (Claiming the groups of a cluster with the same
// weight rows one after the other, as fwd_item orders learners, measured slower: this
// kernel is not bound by DRAM, and the groups' simultaneous reads of the same lines
// cost more than the L2 hits save, 12288-4096-4096-1000 forwards +4 us per launch.)
__device__ __forceinline__ GfItem gf_item(const TcFwdArgs& a, int G, int nk, int it) {
  const int gw = a.n_whole / G;                 // whole group tiles
  GfItem f;
  int gt = it;
  if (it < gw) {
    f.c_lo = 0;
    f.c_hi = nk;
    f.piece = 0;
    f.np = 1;
  } else {
    const int np = a.np_tail, i2 = it - gw, tt = i2 / np, p = i2 - tt * np;
    gt = gw + tt;
    f.c_lo = p * a.piece_chunks;
    f.c_hi = f.c_lo + a.piece_chunks < nk ? f.c_lo + a.piece_chunks : nk;
    f.piece = p;
    f.np = np;
  }
  f.q = gt / a.o_tiles;
  f.ot = gt - f.q * a.o_tiles;
  return f;
}

__global__ void __launch_bounds__(kFwdThreads, 1)
    k_tc_forward_group(const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_h,
                       const TcFwdArgs a, int G) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nk = (a.in + 63) / 64;
  const int N = G * a.Bn;
  const int gtiles = a.n_tiles / G, gw = a.n_whole / G;
  const int n_items = gw + (gtiles - gw) * a.np_tail;
  const int nw = kGfWRing, nh = gf_hring(N);
  const int tbytes = a.Bn * 128, hbytes = N * 128;
  const int h_row0 = a.x_direct ? a.x_row0 : 0;
  uint8_t* h_base = smem + gf_h_off();
  uint64_t* wfull = reinterpret_cast<uint64_t*>(smem + gf_bar_off(N));
  uint64_t* wempty = wfull + kFwdWRingMax;
  uint64_t* hfull = wempty + kFwdWRingMax;
  uint64_t* hempty = hfull + kFwdHRingMax;
  uint64_t* conv = hempty + kFwdHRingMax;  // [kGfABufs] A tile written to TMEM
  uint64_t* wfree = conv + kGfABufs;       // [kGfABufs] A tile consumed by the MMA
  uint64_t* accf = wfree + kGfABufs;       // [2] accumulator segment complete
  uint64_t* accr = accf + 2;               // [2] accumulator segment drained
  uint64_t* gbar = accr + 2;
  uint64_t* done = gbar + 1;
  ItemQueue queue{done + 1, done + 1 + kQueue, nullptr};
  queue.items = reinterpret_cast<int*>(done + 1 + 2 * kQueue);
  int* last_flag = queue.items + kQueue;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(last_flag + 1);
  auto wf = [&](int s) { return smem + s * kFwdWf32; };
  auto hb = [&](int s) { return h_base + s * hbytes; };
  constexpr int kConsumers = 2 + kFwdConv / 32;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kFwdWRingMax; ++s) {
      mbar_init(&wfull[s], 1);
      mbar_init(&wempty[s], kFwdConv / 32);
    }
    for (int s = 0; s < kFwdHRingMax; ++s) {
      mbar_init(&hfull[s], 1);
      mbar_init(&hempty[s], 1);
    }
    for (int b = 0; b < kGfABufs; ++b) {
      mbar_init(&conv[b], kFwdConv / 32);
      mbar_init(&wfree[b], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&accr[b], kFwdConv);
    }
    for (int q = 0; q < kQueue; ++q) {
      mbar_init(&queue.full[q], 1);
      mbar_init(&queue.empty[q], kConsumers);
    }
    mbar_init(gbar, kFwdConv);
    mbar_init(done, 1);
    fence_barrier_init();
  }
  if (warp == 9) {
    tmem_alloc(tmem_slot, kGfTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  grid_dep_wait();

  auto next_item = [&](int k, GfItem& f) -> bool {
    const int it = queue.take(k, lane, a.err);
    if (it < 0) return false;
    f = gf_item(a, G, nk, it);
    return true;
  };

  if (warp == 8) {
    if (lane == 0) {
      // claim, announce, and stream the weight tiles of the cluster mean (normal L2
      // policy: the cluster's other groups read them too)
      tma_prefetch_desc(&tm_w);
      const uint64_t pol = l2_weight_policy(a.w_stream != 0, true);
      int i = 0, issued = 0;
      bool ok = true;
      int next = atomicAdd(a.dyn, 1);
      for (int k = 0; ok; ++k) {
        const int it = next < n_items ? next : -1;
        if (!queue.put(k, it, a.err) || it < 0) break;
        next = atomicAdd(a.dyn, 1);
        const GfItem f = gf_item(a, G, nk, it);
        const int jw = f.q * G / a.w_div;
        for (int c = f.c_lo; c < f.c_hi; ++c, ++i) {
          const int s = i % nw;
          if (i >= nw && !mbar_wait(&wempty[s], ((i / nw) - 1) & 1, a.err)) { ok = false; break; }
          mbar_arrive_expect_tx(&wfull[s], kFwdWf32);
          tma_load_3d_hint(wf(s), &tm_w, &wfull[s], c * 64, f.ot * 128, jw, pol);
          tma_load_3d_hint(wf(s) + kFwdWBox, &tm_w, &wfull[s], c * 64 + 32, f.ot * 128, jw, pol);
          issued = i + 1;
        }
      }
      for (int u = issued - nw > 0 ? issued - nw : 0; u < issued; ++u)
        mbar_wait(&wfull[u % nw], (u / nw) & 1, a.err);
    }
  } else if (warp == 10) {
    // the G learners' batch tiles of each chunk, stacked: learner m's rows at m * Bn
    if (lane == 0) tma_prefetch_desc(&tm_h);
    int i = 0, issued = 0;
    bool ok = true;
    GfItem f;
    for (int k = 0; ok && next_item(k, f); ++k) {
      if (lane == 0) {
        const int j0 = f.q * G;
        for (int c = f.c_lo; c < f.c_hi; ++c, ++i) {
          const int s = i % nh;
          if (i >= nh && !mbar_wait(&hempty[s], ((i / nh) - 1) & 1, a.err)) { ok = false; break; }
          mbar_arrive_expect_tx(&hfull[s], hbytes);
          for (int m = 0; m < G; ++m)
            tma_load_3d(hb(s) + m * tbytes, &tm_h, &hfull[s], c * 64, h_row0, j0 + m);
          issued = i + 1;
        }
      }
      ok = __all_sync(0xffffffffu, ok);
    }
    if (lane == 0)
      for (int u = issued - nh > 0 ? issued - nh : 0; u < issued; ++u)
        mbar_wait(&hfull[u % nh], (u / nh) & 1, a.err);
  } else if (warp == 9) {
    const uint32_t idesc = umma_idesc_bf16(128, N);
    int q = -1, i = 0;
    bool ok = true;
    GfItem f;
    for (int k = 0; ok && next_item(k, f); ++k) {
      if (lane == 0) {
        for (int c = f.c_lo, p = 0; c < f.c_hi; ++c, ++p, ++i) {
          const bool tlast = c == f.c_hi - 1;
          const bool first = p % kSegChunks == 0, last = tlast || p % kSegChunks == kSegChunks - 1;
          const int sh = i % nh, b = i & (kGfABufs - 1);
          if (first) ++q;
          const int ab = q & 1;
          if (first && q >= 2 && !mbar_wait(&accr[ab], ((q >> 1) - 1) & 1, a.err)) { ok = false; break; }
          if (!mbar_wait(&conv[b], (i / kGfABufs) & 1, a.err)) { ok = false; break; }
          if (!mbar_wait(&hfull[sh], (i / nh) & 1, a.err)) { ok = false; break; }
          tc_fence_after();
          const uint32_t at = tmem + kGfTmemA + 32 * b;
          const uint64_t bd = umma_desc_sw128(smem_u32(hb(sh)));
          const uint32_t d = tmem + 128 * ab;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_bf16_ta(d, at + 8 * kk, bd + 2 * kk, idesc, (!first || kk > 0) ? 1u : 0u);
          tc_commit(&hempty[sh]);
          tc_commit(&wfree[b]);
          if (last) tc_commit(&accf[ab]);
        }
      }
      ok = __all_sync(0xffffffffu, ok);
    }
    if (lane == 0) {
      tc_commit(done);
      mbar_wait(done, 0, a.err);
    }
  } else {
    // ---- warps 0-7: fp32 -> bf16 A tile, the accumulator drains and the epilogues.
    // Thread t: accumulator row r (output 128 * ot + r), column blocks 2m + gr of 16
    // (m = 0..3), column = learner (q * G + col / Bn), sample col % Bn.
    const int t = threadIdx.x;
    const int r = t & 127, gr = t >> 7;
    const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
    GroupSync gsync{gbar, 0, a.err};
    float acc[64];
#pragma unroll
    for (int q = 0; q < 64; ++q) acc[q] = 0.f;
    int qc = -1, drained = 0;
    auto drain = [&]() -> bool {
      const int ab = drained & 1;
      if (!wait_warp(&accf[ab], (drained >> 1) & 1, a.err)) return false;
      tc_fence_after();
#pragma unroll
      for (int m = 0; m < 4; ++m) {
        const int cb = (2 * m + gr) * 16;
        if (cb < N) {
          float v[16];
          tmem_ld16(tbase + 128 * ab + cb, v);
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 16; ++q) acc[16 * m + q] = __fadd_rn(acc[16 * m + q], v[q]);
        }
      }
      tc_fence_before();
      mbar_arrive(&accr[ab]);
      ++drained;
      return true;
    };
    auto epilogue = [&](const GfItem& f, float bias) {
      const int o = f.ot * 128 + r;
      if (o >= a.out) return;
#pragma unroll
      for (int m = 0; m < 4; ++m) {
        const int cb = (2 * m + gr) * 16;
        if (cb >= N) break;
        const int ml = cb / a.Bn, b0 = cb - ml * a.Bn;
        const int64_t j = static_cast<int64_t>(f.q) * G + ml;
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          if (b0 + q >= a.B) break;
          if (a.mode == kFwdHidden)
            a.h_out[(j * a.Bn + b0 + q) * a.pitch_out + o] =
                __float2bfloat16_rn(fmaxf(__fadd_rn(acc[16 * m + q], bias), 0.f));
          else
            a.z_out[(j * a.B + b0 + q) * a.out + o] = __fadd_rn(acc[16 * m + q], bias);
        }
      }
    };
    // A tail piece ends: its partials go to the G learners' slots (slot of learner j's
    // tile tau = j * o_tiles + ot, as k_tc_forward's), counted on the first learner's
    // tile; the piece completing the group tile sums every learner's partials in piece
    // order (true: it runs the epilogue).
    auto group_piece_end = [&](const GfItem& f, bool& ok) -> bool {
      const int64_t slot_stride = static_cast<int64_t>(128) * a.Bn;
      auto slot = [&](int ml, int p) {
        const int64_t tt = (static_cast<int64_t>(f.q) * G + ml) * a.o_tiles + f.ot - a.n_whole;
        return a.part + ((tt * f.np + p) * 128 + r) * a.Bn;
      };
#pragma unroll
      for (int m = 0; m < 4; ++m) {
        const int cb = (2 * m + gr) * 16;
        if (cb < N) {
          const int ml = cb / a.Bn, b0 = cb - ml * a.Bn;
          float* dst = slot(ml, f.piece) + b0;
#pragma unroll
          for (int q = 0; q < 16; q += 4)
            __stcg(reinterpret_cast<float4*>(dst + q),
                   make_float4(acc[16 * m + q], acc[16 * m + q + 1], acc[16 * m + q + 2], acc[16 * m + q + 3]));
        }
      }
      if (!gsync()) { ok = false; return false; }
      if (t == 0) {
        const int64_t tt0 = static_cast<int64_t>(f.q) * G * a.o_tiles + f.ot - a.n_whole;
        fence_acq_rel_gpu();
        const int before = atomicAdd(a.counters + tt0, 1);
        const int lastp = before == f.np - 1;
        if (lastp) {
          fence_acq_rel_gpu();
          a.counters[tt0] = 0;
        }
        *last_flag = lastp;
      }
      if (!gsync()) { ok = false; return false; }
      if (!*reinterpret_cast<volatile int*>(last_flag)) return false;
#pragma unroll
      for (int m = 0; m < 4; ++m) {
        const int cb = (2 * m + gr) * 16;
        if (cb < N) {
          const int ml = cb / a.Bn, b0 = cb - ml * a.Bn;
          const float* src = slot(ml, 0) + b0;
#pragma unroll
          for (int q = 0; q < 16; q += 4) {
            float4 s0 = __ldcg(reinterpret_cast<const float4*>(src + q));
            for (int p = 1; p < f.np; ++p) {
              const float4 v = __ldcg(reinterpret_cast<const float4*>(src + p * slot_stride + q));
              s0.x = __fadd_rn(s0.x, v.x);
              s0.y = __fadd_rn(s0.y, v.y);
              s0.z = __fadd_rn(s0.z, v.z);
              s0.w = __fadd_rn(s0.w, v.w);
            }
            acc[16 * m + q] = s0.x;
            acc[16 * m + q + 1] = s0.y;
            acc[16 * m + q + 2] = s0.z;
            acc[16 * m + q + 3] = s0.w;
          }
        }
      }
      return true;
    };
    bool ok = true;
    int i = 0;
    GfItem f;
    for (int k = 0; ok && next_item(k, f); ++k) {
      const int ob = f.ot * 128 + r;
      const float tbias = ob < a.out ? a.bias[static_cast<int64_t>(f.q * G / a.b_div) * a.ld + ob] : 0.f;
      for (int c = f.c_lo, p = 0; c < f.c_hi && ok; ++c, ++p, ++i) {
        const bool tlast = c == f.c_hi - 1;
        const int sw = i % nw, bb = i & (kGfABufs - 1);
        if (!wait_warp(&wfull[sw], (i / nw) & 1, a.err)) { ok = false; break; }
        if (i >= kGfABufs && !wait_warp(&wfree[bb], ((i / kGfABufs) - 1) & 1, a.err)) { ok = false; break; }
        tc_fence_after();
        {
          const int row = 32 * (warp & 3) + lane, half = warp >> 2;
          const uint8_t* src = wf(sw) + half * kFwdWBox + row * 128;
          uint32_t pk[16];
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            const float4 x = *reinterpret_cast<const float4*>(src + ((q ^ (row & 7)) << 4));
            pk[2 * q] = pack_bf16x2(x.x, x.y);
            pk[2 * q + 1] = pack_bf16x2(x.z, x.w);
          }
          tmem_st16(tbase + kGfTmemA + 32 * bb + 16 * half, pk);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&wempty[sw]);
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&conv[bb]);
        if (p % kSegChunks == 0) ++qc;
        if (tlast) {
          while (ok && drained <= qc)
            if (!drain()) ok = false;
          if (!ok) break;
          const bool fin = f.np == 1 || group_piece_end(f, ok);
          if (ok && fin) epilogue(f, tbias);
#pragma unroll
          for (int q = 0; q < 64; ++q) acc[q] = 0.f;
          ok = __all_sync(0xffffffffu, ok);
        } else if (p % kSegChunks == kSegChunks - 1 && qc >= 1 && drained < qc) {
          if (!drain()) ok = false;
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kGfTmemCols);
  }
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(a.dyn + 1, 1) == static_cast<int>(gridDim.x) - 1) {
      a.dyn[0] = 0;
      a.dyn[1] = 0;
    }
  }
}


// ------------------------------------------------------------------ backward
// Backward of one layer on the tensor cores.  Tile = (learner j, input features i0 ..
// i0+127), chunk = output rows o0 .. o0+63 of W_l.  Per chunk:
//   dW^T[i][o] = sum_b H_{l-1}[b][i] dZ_l[b][o]    both operands MN-major, read as stored
//                                                  (H tile of the tile, dZ tile of the chunk)
//   W[o][i]   -= lr dW^T[i][o]                     fp32, in shared memory, then TMA-stored
//   dH^T[i][b] += sum_o W[o][i] dZ_l[b][o]          pre-update weights (A = W^T, bf16, in TMEM)
// so W is read once and written once.  dH^T of a tile accumulates over its chunks (with
// the same every-kSegChunks promotion as the forward), and the tile epilogue applies
// the ReLU mask of H_{l-1}, writes dZ_{l-1} and updates b_{l-1}.  Without dX (the
// first layer) only dW and the update remain.
// The work is claimed dynamically like the forward's: whole tiles, then the last
// tiles (one per SM) split into pieces of TcBwdArgs::piece_chunks chunks; a piece
// writes its dH^T partial to its slot, and the piece that completes a tile adds the
// tile's partials in piece order and runs the epilogue (no CTA waits for another).
// Warps 0-3 and 8-11: the two threads (w % 4, lane) of warps w and w + 8 own input
// feature i0 + 32 (w % 4) + lane (a TMEM lane), each half of the chunk's 64 outputs and
// half of the dH^T columns: they convert their half column of the fp32 chunk to the bf16
// A tile, apply the update in shared memory and promote dH^T; the tile epilogue gathers
// the row in TMEM for one of them.  (With four converter warps, one thread per column,
// the converters set the pace of the pipeline.)  Warp 4 claims the work items and loads
// W chunks and each item's H tile, warp 5 issues the MMAs, warp 6 loads dZ tiles, warp 7
// TMA-stores updated chunks (bulk stores: per-thread row stores of the same bytes ran at
// half the speed) and frees their slots once read.  Each waiting role has a warp of its
// own: a lane blocked in an mbarrier wait holds up the other lanes of its warp.
// (k_tc_update keeps four converter warps, one thread per column, for Q = 1.)
constexpr int kBwdConv = 128;
constexpr int kBwdThreads = kBwdConv + 128;
// k_tc_backward: eight converter warps (0-3 and 8-11), each thread half of a column.
constexpr int kBxConv = 256;
constexpr int kBxThreads = kBxConv + 128;
constexpr int kBwdWf32 = 64 * 128 * 4;                 // 32 KB fp32 W chunk [64 o][128 i]
constexpr int kBwdWRingMax = 5, kBwdZRingMax = 8;
constexpr int kBwdSmemMax = 227 * 1024;
// TMEM columns: dH^T accumulators at 0 and 64, dW^T at 128 and 192, W^T (A) at 256, 288,
// and (k_tc_backward) the tile's promoted dH^T gathered for its epilogue at 320.
constexpr uint32_t kBwdTmemCols = 512;
constexpr uint32_t kBwdTmemW = 128, kBwdTmemA = 256, kBwdTmemS = 320;

// Layout: W ring | 2 H tiles (2 x [Bn][64] bf16 each) | dZ ring ([Bn][64] bf16) | barriers.
__host__ __device__ constexpr int bwd_wring(int Bn) { return (void)Bn, 5; }
__host__ __device__ constexpr int bwd_h_off(int Bn) { return bwd_wring(Bn) * kBwdWf32; }
__host__ __device__ constexpr int bwd_z_off(int Bn) { return bwd_h_off(Bn) + 2 * 2 * Bn * 128; }
__host__ __device__ constexpr int bwd_zring(int Bn) {
  return (kBwdSmemMax - 1024 - kBarBytes - bwd_z_off(Bn)) / (Bn * 128) < kBwdZRingMax
             ? (kBwdSmemMax - 1024 - kBarBytes - bwd_z_off(Bn)) / (Bn * 128)
             : kBwdZRingMax;
}
__host__ __device__ constexpr int bwd_bar_off(int Bn) { return bwd_z_off(Bn) + bwd_zring(Bn) * Bn * 128; }
__host__ __device__ constexpr int bwd_smem(int Bn) { return bwd_bar_off(Bn) + kBarBytes + 1024; }
static_assert(bwd_zring(64) >= 4 && bwd_zring(48) >= 6 && bwd_zring(32) >= 8 && bwd_zring(16) >= 8 &&
                  bwd_smem(64) <= kBwdSmemMax && bwd_smem(48) <= kBwdSmemMax &&
                  bwd_smem(32) <= kBwdSmemMax && bwd_smem(16) <= kBwdSmemMax,
              "backward shared-memory plan");

// kNoUpd: dZ_{l-1} and b_{l-1} only (TcBwdArgs::no_update), compiled separately so that
// the full backward carries none of its branches.
template <bool kNoUpd>
__global__ void __launch_bounds__(kBxThreads, 1)
    k_tc_backward(const __grid_constant__ CUtensorMap tm_wl, const __grid_constant__ CUtensorMap tm_ws,
                  const __grid_constant__ CUtensorMap tm_h, const __grid_constant__ CUtensorMap tm_dz,
                  const TcBwdArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nc = (a.out + 63) / 64;
  const int n_items = a.n_whole + (a.n_tiles - a.n_whole) * a.np_tail;
  const int nw = bwd_wring(a.Bn), nz = bwd_zring(a.Bn);
  const int tbytes = a.Bn * 128;                           // one [Bn][64] bf16 tile
  uint8_t* h_base = smem + bwd_h_off(a.Bn);
  uint8_t* z_base = smem + bwd_z_off(a.Bn);
  uint64_t* wfull = reinterpret_cast<uint64_t*>(smem + bwd_bar_off(a.Bn));
  uint64_t* wempty = wfull + kBwdWRingMax;   // chunk stored back (TMA has read it)
  uint64_t* upd = wempty + kBwdWRingMax;     // chunk updated in shared memory
  uint64_t* zfull = upd + kBwdWRingMax;
  uint64_t* zempty = zfull + kBwdZRingMax;   // dZ tile consumed by both MMAs
  uint64_t* hfull = zempty + kBwdZRingMax;   // [2]
  uint64_t* hempty = hfull + 2;              // [2] the item's epilogue (or last MMA) is done
  uint64_t* conv = hempty + 2;               // [2] W^T written to TMEM
  uint64_t* afree = conv + 2;                // [2] W^T consumed by the dX MMA
  uint64_t* dwdone = afree + 2;              // [2] dW^T of the chunk complete
  uint64_t* dwfree = dwdone + 2;             // [2] dW^T read by the update
  uint64_t* xf = dwfree + 2;                 // [2] dH^T segment complete
  uint64_t* xr = xf + 2;                     // [2] dH^T segment drained
  uint64_t* gbar = xr + 2;
  uint64_t* done = gbar + 1;
  ItemQueue queue{done + 1, done + 1 + kQueue, nullptr};
  queue.items = reinterpret_cast<int*>(done + 1 + 2 * kQueue);
  int* last_flag = queue.items + kQueue;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(last_flag + 1);
  auto wf = [&](int s) { return smem + s * kBwdWf32; };
  auto hb = [&](int s) { return h_base + s * 2 * tbytes; };
  auto zb = [&](int s) { return z_base + s * tbytes; };
  constexpr int kConsumers = 3 + kBxConv / 32;              // MMA, dZ, store + converter warps

  if (threadIdx.x == 0) {
    for (int s = 0; s < kBwdWRingMax; ++s) {
      mbar_init(&wfull[s], 1);
      mbar_init(&wempty[s], 1);
      mbar_init(&upd[s], kBxConv / 32);
    }
    for (int s = 0; s < kBwdZRingMax; ++s) {
      mbar_init(&zfull[s], 1);
      mbar_init(&zempty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&hfull[b], 1);
      mbar_init(&hempty[b], kBxConv / 32);
      mbar_init(&conv[b], kBxConv / 32);
      mbar_init(&afree[b], 1);
      mbar_init(&dwdone[b], 1);
      mbar_init(&dwfree[b], kBxConv / 32);
      mbar_init(&xf[b], 1);
      mbar_init(&xr[b], kBxConv / 32);
    }
    for (int q = 0; q < kQueue; ++q) {
      mbar_init(&queue.full[q], 1);
      mbar_init(&queue.empty[q], kConsumers);
    }
    mbar_init(gbar, kBxConv);
    mbar_init(done, 1);
    fence_barrier_init();
  }
  if (warp == 5) {
    tmem_alloc(tmem_slot, kBwdTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  grid_dep_wait();                       // the previous kernel's results are visible

  auto next_item = [&](int k, FwdItem& f) -> bool {
    const int it = queue.take(k, lane, a.err);
    if (it < 0) return false;
    f = fwd_item(a, nc, it);
    return true;
  };

  if (warp == 4) {
    if (lane == 0) {
      // claim, announce, and load: each item's H tile (two 64-feature boxes) ahead of
      // its first W chunk, then its W chunks
      tma_prefetch_desc(&tm_wl);
      tma_prefetch_desc(&tm_h);
      const uint64_t stream = l2_weight_policy(a.w_stream != 0, a.src_div > 1);
      int i = 0, issued = 0;
      bool ok = true;
      int next = atomicAdd(a.dyn, 1);
      for (int k = 0; ok; ++k) {
        const int it = next < n_items ? next : -1;
        if (!queue.put(k, it, a.err) || it < 0) break;
        next = atomicAdd(a.dyn, 1);           // the next claim, hidden behind these loads
        const FwdItem f = fwd_item(a, nc, it);
        const int j = f.tau / a.s_tiles, i0 = (f.tau - j * a.s_tiles) * 128;
        const int hbuf = k & 1;
        if (k >= 2 && !mbar_wait(&hempty[hbuf], ((k >> 1) - 1) & 1, a.err)) break;
        mbar_arrive_expect_tx(&hfull[hbuf], 2 * tbytes);
        tma_load_3d(hb(hbuf), &tm_h, &hfull[hbuf], i0, a.h_row0, j);
        tma_load_3d(hb(hbuf) + tbytes, &tm_h, &hfull[hbuf], i0 + 64, a.h_row0, j);
        for (int c = f.c_lo; c < f.c_hi; ++c, ++i) {
          const int s = i % nw;
          if (i >= nw && !mbar_wait(&wempty[s], ((i / nw) - 1) & 1, a.err)) { ok = false; break; }
          mbar_arrive_expect_tx(&wfull[s], kBwdWf32);
          tma_load_3d_hint(wf(s), &tm_wl, &wfull[s], i0, c * 64, j / a.src_div, stream);
          issued = i + 1;
        }
      }
      for (int u = issued - nw > 0 ? issued - nw : 0; u < issued; ++u)
        mbar_wait(&wfull[u % nw], (u / nw) & 1, a.err);
    }
  } else if (warp == 6) {
    // dZ tiles of each chunk
    if (lane == 0) tma_prefetch_desc(&tm_dz);
    int i = 0, issued = 0;
    bool ok = true;
    FwdItem f;
    for (int k = 0; ok && next_item(k, f); ++k) {
      if (lane == 0) {
        const int j = f.tau / a.s_tiles;
        for (int c = f.c_lo; c < f.c_hi; ++c, ++i) {
          const int s = i % nz;
          if (i >= nz && !mbar_wait(&zempty[s], ((i / nz) - 1) & 1, a.err)) { ok = false; break; }
          mbar_arrive_expect_tx(&zfull[s], tbytes);
          tma_load_3d(zb(s), &tm_dz, &zfull[s], c * 64, 0, j);
          issued = i + 1;
        }
      }
      ok = __all_sync(0xffffffffu, ok);
    }
    if (lane == 0)
      for (int u = issued - nz > 0 ? issued - nz : 0; u < issued; ++u)
        mbar_wait(&zfull[u % nz], (u / nz) & 1, a.err);
  } else if (warp == 7) {
    // Store each updated chunk; its slot is released once the TMA has read it (two
    // stores in flight; when the chunks come from the cluster means, as soon as its own
    // store has been read).  no_update: the slot is released as soon as it has been read.
    const uint64_t stream = l2_weight_policy(a.w_stream != 0);
    const bool store = !kNoUpd, eager = a.src_div > 1;
    int i = 0, released = 0;
    bool ok = true;
    FwdItem f;
    for (int k = 0; ok && next_item(k, f); ++k) {
      if (lane == 0) {
        const int j = f.tau / a.s_tiles, i0 = (f.tau - j * a.s_tiles) * 128;
        for (int c = f.c_lo; c < f.c_hi; ++c, ++i) {
          const int s = i % nw;
          if (!mbar_wait(&upd[s], (i / nw) & 1, a.err)) { ok = false; break; }
          if (!store) {
            mbar_arrive(&wempty[s]);
            continue;
          }
          tma_store_3d_hint(&tm_ws, wf(s), i0, c * 64, j, stream);
          tma_store_commit();
          if (eager) {
            tma_store_wait_read_all();
            mbar_arrive(&wempty[s]);
            released = i + 1;
          } else if (i > 0) {
            tma_store_wait_read_1();
            mbar_arrive(&wempty[(i - 1) % nw]);
            released = i;
          }
        }
      }
      ok = __all_sync(0xffffffffu, ok);
    }
    if (lane == 0 && store) {
      tma_store_wait_read_all();   // (before the shared memory is released)
      if (i > released) mbar_arrive(&wempty[(i - 1) % nw]);
    }
  } else if (warp == 5) {
    const uint32_t idesc_dw = umma_idesc_bf16(128, 64) | (1u << 15) | (1u << 16);
    const uint32_t idesc_dx = umma_idesc_bf16(128, a.Bn);
    const int kb = a.Bn / 16;   // K = Bn for dW
    int i = 0, q = -1;
    bool ok = true;
    FwdItem f;
    for (int k = 0; ok && next_item(k, f); ++k) {
      if (lane == 0) {
        if (!mbar_wait(&hfull[k & 1], (k >> 1) & 1, a.err)) ok = false;
        const uint32_t hs = smem_u32(hb(k & 1));
        for (int c = f.c_lo, p = 0; ok && c < f.c_hi; ++c, ++p, ++i) {
          const bool tlast = c == f.c_hi - 1;
          const bool first = p % kSegChunks == 0, last = tlast || p % kSegChunks == kSegChunks - 1;
          const int sz = i % nz, b = i & 1;
          if (!mbar_wait(&zfull[sz], (i / nz) & 1, a.err)) { ok = false; break; }
          const uint32_t zs = smem_u32(zb(sz));
          if constexpr (!kNoUpd) {
            if (i >= 2 && !mbar_wait(&dwfree[b], ((i >> 1) - 1) & 1, a.err)) { ok = false; break; }
            tc_fence_after();
            for (int kk = 0; kk < kb; ++kk)
              tc_mma_bf16(tmem + kBwdTmemW + 64 * b, umma_desc_sw128_mn(hs + kk * 2048, tbytes),
                          umma_desc_sw128_mn(zs + kk * 2048, tbytes), idesc_dw, kk > 0 ? 1u : 0u);
            tc_commit(&dwdone[b]);
          }
          if (a.has_dx) {
            if (first) ++q;
            const int xb = q & 1;
            if (first && q >= 2 && !mbar_wait(&xr[xb], ((q >> 1) - 1) & 1, a.err)) { ok = false; break; }
            if (!mbar_wait(&conv[b], (i >> 1) & 1, a.err)) { ok = false; break; }
            tc_fence_after();
            const uint64_t zd = umma_desc_sw128(zs);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc_mma_bf16_ta(tmem + 64 * xb, tmem + kBwdTmemA + 32 * b + 8 * kk, zd + 2 * kk, idesc_dx,
                             (!first || kk > 0) ? 1u : 0u);
            tc_commit(&afree[b]);
            if (last) tc_commit(&xf[xb]);
          }
          tc_commit(&zempty[sz]);
        }
      }
      ok = __all_sync(0xffffffffu, ok);
    }
    if (lane == 0) {
      tc_commit(done);
      mbar_wait(done, 0, a.err);
    }
  } else {
    // ---- warps 0-3 and 8-11: thread (warp % 4, lane) owns input feature i0 + t of the
    // tile (TMEM lane t); warps 0-3 outputs 0-31 of each chunk and the dH^T column blocks
    // 0 and 2 (16 samples each), warps 8-11 outputs 32-63 and blocks 1 and 3
    const int t = 32 * (warp & 3) + lane, hf = warp >= 8 ? 1 : 0, o0 = 32 * hf;
    const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
    GroupSync gsync{gbar, 0, a.err};
    float accx[32];                                // dH^T[i0 + t][16 (2m + hf) + q], promoted
#pragma unroll
    for (int q = 0; q < 32; ++q) accx[q] = 0.f;
    int qc = -1, drained = 0;
    auto drain = [&]() -> bool {
      const int xb = drained & 1;
      if (!wait_warp(&xf[xb], (drained >> 1) & 1, a.err)) return false;
      tc_fence_after();
#pragma unroll
      for (int m = 0; m < 2; ++m) {
        const int cb = 16 * (2 * m + hf);
        if (cb < a.Bn) {
          float v[16];
          tmem_ld16(tbase + 64 * xb + cb, v);
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 16; ++q) accx[16 * m + q] = __fadd_rn(accx[16 * m + q], v[q]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&xr[xb]);
      ++drained;
      return true;
    };
    // A split tile's piece ends: this thread's blocks go to the piece's slot (slot (tail
    // tile tt, piece p) = part[((tt * np + p) * 128 + t) * Bn]); the piece completing the
    // tile replaces them with the sums of the tile's partials in piece order.
    auto piece_end = [&](const FwdItem& f, bool& ok) -> bool {
      const int tt = f.tau - a.n_whole;
      const int64_t pstride = static_cast<int64_t>(128) * a.Bn;
      float* mine = a.part + (static_cast<int64_t>(tt) * f.np + f.piece) * pstride +
                    static_cast<int64_t>(t) * a.Bn;
#pragma unroll
      for (int m = 0; m < 2; ++m) {
        const int cb = 16 * (2 * m + hf);
        if (cb < a.Bn) {
#pragma unroll
          for (int q = 0; q < 16; q += 4)
            __stcg(reinterpret_cast<float4*>(mine + cb + q),
                   make_float4(accx[16 * m + q], accx[16 * m + q + 1], accx[16 * m + q + 2],
                               accx[16 * m + q + 3]));
        }
      }
      if (!gsync()) { ok = false; return false; }
      if (threadIdx.x == 0) {
        fence_acq_rel_gpu();
        const int before = atomicAdd(a.counters + tt, 1);
        const int last = before == f.np - 1;
        if (last) {
          fence_acq_rel_gpu();
          a.counters[tt] = 0;
        }
        *last_flag = last;
      }
      if (!gsync()) { ok = false; return false; }
      if (!*reinterpret_cast<volatile int*>(last_flag)) return false;
      const float* src = a.part + static_cast<int64_t>(tt) * f.np * pstride + static_cast<int64_t>(t) * a.Bn;
#pragma unroll
      for (int m = 0; m < 2; ++m) {
        const int cb = 16 * (2 * m + hf);
        if (cb >= a.Bn) continue;
#pragma unroll
        for (int q = 0; q < 16; q += 4) {
          float4 s0 = __ldcg(reinterpret_cast<const float4*>(src + cb + q));
          for (int p = 1; p < f.np; ++p) {
            const float4 v = __ldcg(reinterpret_cast<const float4*>(src + p * pstride + cb + q));
            s0.x = __fadd_rn(s0.x, v.x);
            s0.y = __fadd_rn(s0.y, v.y);
            s0.z = __fadd_rn(s0.z, v.z);
            s0.w = __fadd_rn(s0.w, v.w);
          }
          accx[16 * m + q] = s0.x;
          accx[16 * m + q + 1] = s0.y;
          accx[16 * m + q + 2] = s0.z;
          accx[16 * m + q + 3] = s0.w;
        }
      }
      return true;
    };
    // dZ_{l-1}[b][i] = dH[b][i] * (H_{l-1}[b][i] > 0), b < B; b_{l-1}[i] -= lr sum_b.  The
    // row's blocks are gathered in TMEM, so that one thread adds the bias gradient in
    // sample order.  (The item's H tile landed long ago; the wait makes the TMA's writes
    // visible here.)
    auto epilogue = [&](int tau, int k) -> bool {
#pragma unroll
      for (int m = 0; m < 2; ++m) {
        const int cb = 16 * (2 * m + hf);
        if (cb < a.Bn) {
          uint32_t r[16];
#pragma unroll
          for (int q = 0; q < 16; ++q) r[q] = __float_as_uint(accx[16 * m + q]);
          tmem_st16(tbase + kBwdTmemS + cb, r);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      if (!gsync()) return false;
      tc_fence_after();
      if (!wait_warp(&hfull[k & 1], (k >> 1) & 1, a.err)) return false;
      const int j = tau / a.s_tiles, fi = (tau - j * a.s_tiles) * 128 + t;
      if (hf == 0) {
        float db = 0.f;
        const uint8_t* hcol = hb(k & 1) + (t >> 6) * a.Bn * 128;
        __nv_bfloat16* dz = a.dz_prev + static_cast<int64_t>(j) * a.Bn * a.pitch_in + fi;
#pragma unroll
        for (int cb = 0; cb < 64; cb += 16) {
          if (cb < a.Bn) {
            float v[16];
            tmem_ld16(tbase + kBwdTmemS + cb, v);
            tmem_ld_wait();
            if (fi < a.in) {
#pragma unroll
              for (int q = 0; q < 16; ++q) {
                const int b = cb + q;
                if (b < a.B) {
                  const __nv_bfloat16 hv =
                      *reinterpret_cast<const __nv_bfloat16*>(hcol + sw128_offset(b, t & 63));
                  const float x = __bfloat162float(hv) > 0.f ? v[q] : 0.f;
                  db = __fadd_rn(db, x);
                  dz[static_cast<int64_t>(b) * a.pitch_in] = __float2bfloat16_rn(x);
                }
              }
            }
          }
        }
        if (fi < a.in) {
          const float bv = a.bias_prev_src[static_cast<int64_t>(j / a.src_div) * a.ld + fi];
          a.bias_prev[static_cast<int64_t>(j) * a.ld + fi] = __fsub_rn(bv, __fmul_rn(a.lr, db));
        }
      }
      tc_fence_before();
      return gsync();   // the gathered blocks are read before the next tile writes them
    };
    bool ok = true;
    int i = 0;
    FwdItem f;
    for (int k = 0; ok && next_item(k, f); ++k) {
      for (int c = f.c_lo, p = 0; ok && c < f.c_hi; ++c, ++p, ++i) {
        const bool tlast = c == f.c_hi - 1;
        const int sw = i % nw, b = i & 1;
        if (!wait_warp(&wfull[sw], (i / nw) & 1, a.err)) { ok = false; break; }
        float* w = reinterpret_cast<float*>(wf(sw)) + o0 * 128;
        float wv[32];
#pragma unroll
        for (int o = 0; o < 32; ++o) wv[o] = w[o * 128 + t];
        if (a.has_dx) {
          if (i >= 2 && !wait_warp(&afree[b], ((i >> 1) - 1) & 1, a.err)) { ok = false; break; }
          tc_fence_after();
          uint32_t pk[16];
#pragma unroll
          for (int q = 0; q < 16; ++q) pk[q] = pack_bf16x2(wv[2 * q], wv[2 * q + 1]);
          tmem_st16(tbase + kBwdTmemA + 32 * b + 16 * hf, pk);
          tmem_st_wait();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&conv[b]);
        }
        if constexpr (!kNoUpd) {
          if (!wait_warp(&dwdone[b], (i >> 1) & 1, a.err)) { ok = false; break; }
          tc_fence_after();
#pragma unroll
          for (int qb = 0; qb < 2; ++qb) {
            float d[16];
            tmem_ld16(tbase + kBwdTmemW + 64 * b + o0 + 16 * qb, d);
            tmem_ld_wait();
#pragma unroll
            for (int q = 0; q < 16; ++q) wv[16 * qb + q] = __fsub_rn(wv[16 * qb + q], __fmul_rn(a.lr, d[q]));
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&dwfree[b]);
#pragma unroll
          for (int o = 0; o < 32; ++o) w[o * 128 + t] = wv[o];
          fence_proxy_async_smem();
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&upd[sw]);
        if (a.has_dx) {
          if (p % kSegChunks == 0) ++qc;
          if (tlast) {
            while (ok && drained <= qc)
              if (!drain()) ok = false;
            if (ok) {
              const bool fin = f.np == 1 || piece_end(f, ok);
              if (ok && fin && !epilogue(f.tau, k)) ok = false;
              ok = __all_sync(0xffffffffu, ok);
#pragma unroll
              for (int q = 0; q < 32; ++q) accx[q] = 0.f;
            }
          } else if (p % kSegChunks == kSegChunks - 1 && qc >= 1 && drained < qc) {
            if (!drain()) ok = false;
          }
        }
        if (tlast) {
          __syncwarp();
          if (lane == 0) mbar_arrive(&hempty[k & 1]);   // the H tile may be replaced
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kBwdTmemCols);
  }
  if (threadIdx.x == 0) {
    // the last CTA out resets the claim counters for the next launch
    __threadfence();
    if (atomicAdd(a.dyn + 1, 1) == static_cast<int>(gridDim.x) - 1) {
      a.dyn[0] = 0;
      a.dyn[1] = 0;
    }
  }
}

// ------------------------------------------------------------------ update only
// The first layer's backward has no dX: every unit (tile, chunk) is independent
// (dW^T of the chunk, the fp32 update, the store), so the units are handed out
// dynamically and faster SMs simply take more of them (a static split left SMs idle
// for up to a third of the kernel waiting for slow ones).  Work item = a run of up to
// kRun chunks of one tile, claimed by warp 4 from a global counter and announced to
// the other roles through a small queue in shared memory; the last CTA to finish
// resets the counters.  Roles as in k_tc_backward, without the dX path.
//
// Q > 1 (the step that closes a local block, followed by a compact local average): a
// work item covers the same tile and chunks of Q consecutive learners of a cluster
// (learners q*Q .. q*Q+Q-1).  Each learner's updated chunk is formed as for Q = 1, and
// the converter threads add the Q of them in the first log2(Q) levels of the
// adjacent-pair tree of the local average ((w0 + w1) for Q = 2; (w0 + w1) + (w2 + w3)
// for Q = 4), so that only this group sum is stored, to row q of the group-sum buffer
// (store map) instead of Q learner rows.  The local average finishes the tree from
// the group sums: the bits of the literal update and average.
constexpr int kRun = 8;                 // chunks per work item
__host__ __device__ constexpr int upd_smem(int Bn) { return bwd_smem(Bn) + 512; }
static_assert(upd_smem(64) <= kBwdSmemMax && upd_smem(48) <= kBwdSmemMax &&
                  upd_smem(32) <= kBwdSmemMax && upd_smem(16) <= kBwdSmemMax,
              "update kernel shared-memory plan");
// Group layout (Q > 1): W ring (4 slots) | 2 x Q H tiles | dZ ring | barriers and queue.
__host__ __device__ constexpr int updg_h_off(int Q, int Bn) { return (void)Q, (void)Bn, 4 * kBwdWf32; }
__host__ __device__ constexpr int updg_z_off(int Q, int Bn) { return updg_h_off(Q, Bn) + 2 * Q * 2 * Bn * 128; }
__host__ __device__ constexpr int updg_zring(int Q, int Bn) {
  return (kBwdSmemMax - 1024 - kBarBytes - updg_z_off(Q, Bn)) / (Bn * 128) < kBwdZRingMax
             ? (kBwdSmemMax - 1024 - kBarBytes - updg_z_off(Q, Bn)) / (Bn * 128)
             : kBwdZRingMax;
}
__host__ __device__ constexpr int updg_bar_off(int Q, int Bn) {
  return updg_z_off(Q, Bn) + updg_zring(Q, Bn) * Bn * 128;
}
__host__ __device__ constexpr int updg_smem(int Q, int Bn) { return updg_bar_off(Q, Bn) + kBarBytes + 1024; }
static_assert(updg_zring(4, 32) >= 4 && updg_smem(4, 32) <= kBwdSmemMax && updg_zring(4, 16) >= 4 &&
                  updg_smem(4, 16) <= kBwdSmemMax && updg_zring(2, 64) >= 4 &&
                  updg_smem(2, 64) <= kBwdSmemMax && updg_zring(2, 48) >= 4 &&
                  updg_smem(2, 48) <= kBwdSmemMax,
              "group update kernel shared-memory plan");

// Q > 1: eight converter warps (0-3 and 8-11), each thread half of a column.
__host__ __device__ constexpr int upd_conv_warps(int Q) { return Q == 1 ? kBwdConv / 32 : 8; }
__host__ __device__ constexpr int upd_threads(int Q) { return 128 + 32 * upd_conv_warps(Q); }

template <int Q>
__global__ void __launch_bounds__(upd_threads(Q), 1)
    k_tc_update(const __grid_constant__ CUtensorMap tm_wl, const __grid_constant__ CUtensorMap tm_ws,
                const __grid_constant__ CUtensorMap tm_h, const __grid_constant__ CUtensorMap tm_dz,
                const TcBwdArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kChunks = a.run;                               // chunks per item and learner
  const int nc = (a.out + 63) / 64;
  const int rpt = (nc + kChunks - 1) / kChunks;            // work items per tile
  const int n_items = a.n_tiles / Q * rpt;                 // tiles of learner groups
  const int nw = Q == 1 ? bwd_wring(a.Bn) : 4;
  const int nz = Q == 1 ? bwd_zring(a.Bn) : updg_zring(Q, a.Bn);
  const int tbytes = a.Bn * 128;
  uint8_t* h_base = smem + (Q == 1 ? bwd_h_off(a.Bn) : updg_h_off(Q, a.Bn));
  uint8_t* z_base = smem + (Q == 1 ? bwd_z_off(a.Bn) : updg_z_off(Q, a.Bn));
  uint8_t* bar_base = smem + (Q == 1 ? bwd_bar_off(a.Bn) : updg_bar_off(Q, a.Bn));
  uint64_t* wfull = reinterpret_cast<uint64_t*>(bar_base);
  uint64_t* wempty = wfull + kBwdWRingMax;   // chunk stored back (TMA has read it)
  uint64_t* upd = wempty + kBwdWRingMax;     // chunk updated (or read) in shared memory
  uint64_t* zfull = upd + kBwdWRingMax;
  uint64_t* zempty = zfull + kBwdZRingMax;   // dZ tile consumed by the MMA
  uint64_t* hfull = zempty + kBwdZRingMax;   // [2]
  uint64_t* hempty = hfull + 2;              // [2] the item's last MMA is done
  uint64_t* dwdone = hempty + 2;             // [2]
  uint64_t* dwfree = dwdone + 2;             // [2]
  uint64_t* done = dwfree + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  uint64_t* qfull = reinterpret_cast<uint64_t*>(bar_base + 512);
  uint64_t* qempty = qfull + kQueue;         // read by the 7 consuming warps
  int* items = reinterpret_cast<int*>(qempty + kQueue);
  auto wf = [&](int s) { return smem + s * kBwdWf32; };
  // member m's H tile (two 64-feature boxes) in buffer hbuf
  auto hb = [&](int hbuf, int m) { return h_base + (hbuf * Q + m) * 2 * tbytes; };
  auto zb = [&](int s) { return z_base + s * tbytes; };
  constexpr int kConv = upd_conv_warps(Q);
  constexpr int kConsumers = 3 + kConv;                     // dZ, MMA, store + converter warps

  if (threadIdx.x == 0) {
    for (int s = 0; s < kBwdWRingMax; ++s) {
      mbar_init(&wfull[s], 1);
      mbar_init(&wempty[s], 1);
      mbar_init(&upd[s], kConv);
    }
    for (int s = 0; s < kBwdZRingMax; ++s) {
      mbar_init(&zfull[s], 1);
      mbar_init(&zempty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&hfull[b], 1);
      mbar_init(&hempty[b], 1);
      mbar_init(&dwdone[b], 1);
      mbar_init(&dwfree[b], kConv);
    }
    for (int q = 0; q < kQueue; ++q) {
      mbar_init(&qfull[q], 1);
      mbar_init(&qempty[q], kConsumers);
    }
    mbar_init(done, 1);
    fence_barrier_init();
  }
  if (warp == 5) {
    tmem_alloc(tmem_slot, kBwdTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  grid_dep_wait();                       // the previous kernel's results are visible

  // Consumers: the k-th queued work item (-1: no more), read by every lane of the
  // warp; lane 0 then frees the slot for this warp.
  auto take = [&](int k) -> int {
    const int q = k % kQueue;
    if (!wait_warp(&qfull[q], (k / kQueue) & 1, a.err)) return -1;
    const int it = items[q];
    __syncwarp();
    if (lane == 0) mbar_arrive(&qempty[q]);
    return it;
  };
  // Group tile `tile` (group tile / s_tiles, input features 128 * (tile % s_tiles) ..)
  // and its chunks [c_lo, c_hi) for work item `it`.
  auto decode = [&](int it, int& tile, int& c_lo, int& c_hi) {
    tile = it / rpt;
    c_lo = (it - tile * rpt) * kChunks;
    c_hi = c_lo + kChunks < nc ? c_lo + kChunks : nc;
  };

  if (warp == 4) {
    if (lane == 0) {
      // claim, announce, and load: each item's H tiles, then per chunk the W chunks of
      // the group's learners in order
      tma_prefetch_desc(&tm_wl);
      tma_prefetch_desc(&tm_h);
      const uint64_t stream = l2_weight_policy(a.w_stream != 0);
      int i = 0, kt = 0, issued = 0;
      bool ok = true;
      int next = atomicAdd(a.dyn, 1);
      for (int k = 0; ok; ++k) {
        const int it = next < n_items ? next : -1;
        const int q = k % kQueue;
        if (k >= kQueue && !mbar_wait(&qempty[q], ((k / kQueue) - 1) & 1, a.err)) break;
        items[q] = it;
        mbar_arrive(&qfull[q]);
        if (it < 0) break;
        next = atomicAdd(a.dyn, 1);           // the next claim, hidden behind these loads
        int tile, c_lo, c_hi;
        decode(it, tile, c_lo, c_hi);
        const int g = tile / a.s_tiles, i0 = (tile - g * a.s_tiles) * 128, j0 = g * Q;
        const int hbuf = kt & 1;
        if (kt >= 2 && !mbar_wait(&hempty[hbuf], ((kt >> 1) - 1) & 1, a.err)) break;
        mbar_arrive_expect_tx(&hfull[hbuf], Q * 2 * tbytes);
        for (int m = 0; m < Q; ++m) {
          tma_load_3d(hb(hbuf, m), &tm_h, &hfull[hbuf], i0, a.h_row0, j0 + m);
          tma_load_3d(hb(hbuf, m) + tbytes, &tm_h, &hfull[hbuf], i0 + 64, a.h_row0, j0 + m);
        }
        ++kt;
        for (int c = c_lo; c < c_hi && ok; ++c) {
          for (int m = 0; m < Q; ++m, ++i) {
            const int s = i % nw;
            if (i >= nw && !mbar_wait(&wempty[s], ((i / nw) - 1) & 1, a.err)) { ok = false; break; }
            mbar_arrive_expect_tx(&wfull[s], kBwdWf32);
            tma_load_3d_hint(wf(s), &tm_wl, &wfull[s], i0, c * 64, (j0 + m) / a.src_div, stream);
            issued = i + 1;
          }
        }
      }
      for (int u = issued - nw > 0 ? issued - nw : 0; u < issued; ++u)
        mbar_wait(&wfull[u % nw], (u / nw) & 1, a.err);
      for (int u = kt - 2 > 0 ? kt - 2 : 0; u < kt; ++u) mbar_wait(&hfull[u & 1], (u >> 1) & 1, a.err);
    }
  } else if (warp == 6) {
    int i = 0, issued = 0;
    if (lane == 0) tma_prefetch_desc(&tm_dz);
    for (int k = 0;; ++k) {
      const int it = take(k);
      if (it < 0) break;
      if (lane == 0) {
        int tile, c_lo, c_hi;
        decode(it, tile, c_lo, c_hi);
        const int j0 = tile / a.s_tiles * Q;
        bool ok = true;
        for (int c = c_lo; c < c_hi && ok; ++c) {
          for (int m = 0; m < Q; ++m, ++i) {
            const int s = i % nz;
            if (i >= nz && !mbar_wait(&zempty[s], ((i / nz) - 1) & 1, a.err)) { ok = false; break; }
            mbar_arrive_expect_tx(&zfull[s], tbytes);
            tma_load_3d(zb(s), &tm_dz, &zfull[s], c * 64, 0, j0 + m);
            issued = i + 1;
          }
        }
      }
      __syncwarp();
    }
    if (lane == 0)
      for (int u = issued - nz > 0 ? issued - nz : 0; u < issued; ++u)
        mbar_wait(&zfull[u % nz], (u / nz) & 1, a.err);
  } else if (warp == 7) {
    // Q = 1: store each updated chunk, freeing its slot one store behind.  Q > 1: free
    // the slots of the first Q - 1 learners as soon as they are read, store the group
    // sum (row g of the store map) and free its slot once the store has read it.
    const uint64_t stream = l2_weight_policy(a.w_stream != 0);
    int i = 0;
    for (int k = 0;; ++k) {
      const int it = take(k);
      if (it < 0) break;
      if (lane == 0) {
        int tile, c_lo, c_hi;
        decode(it, tile, c_lo, c_hi);
        const int g = tile / a.s_tiles, i0 = (tile - g * a.s_tiles) * 128;
        bool ok = true;
        for (int c = c_lo; c < c_hi && ok; ++c) {
          for (int m = 0; m < Q; ++m, ++i) {
            const int s = i % nw;
            if (!mbar_wait(&upd[s], (i / nw) & 1, a.err)) { ok = false; break; }
            if constexpr (Q == 1) {
              tma_store_3d_hint(&tm_ws, wf(s), i0, c * 64, g, stream);
              tma_store_commit();
              if (i > 0) {
                tma_store_wait_read_1();
                mbar_arrive(&wempty[(i - 1) % nw]);
              }
            } else if (m + 1 < Q) {
              mbar_arrive(&wempty[s]);
            } else {
              tma_store_3d_hint(&tm_ws, wf(s), i0, c * 64, g, stream);
              tma_store_commit();
              tma_store_wait_read_all();
              mbar_arrive(&wempty[s]);
            }
          }
        }
      }
      __syncwarp();
    }
    if (lane == 0) {
      tma_store_wait_read_all();   // (before the shared memory is released)
      if (Q == 1 && i > 0) mbar_arrive(&wempty[(i - 1) % nw]);
    }
  } else if (warp == 5) {
    const uint32_t idesc_dw = umma_idesc_bf16(128, 64) | (1u << 15) | (1u << 16);
    const int kb = a.Bn / 16;
    int i = 0, kt = -1;
    bool ok = true;
    for (int k = 0; ok; ++k) {
      const int it = take(k);
      if (it < 0) break;
      ++kt;
      if (lane == 0) {
        int tile, c_lo, c_hi;
        decode(it, tile, c_lo, c_hi);
        if (!mbar_wait(&hfull[kt & 1], (kt >> 1) & 1, a.err)) ok = false;
        for (int c = c_lo; c < c_hi && ok; ++c) {
          for (int m = 0; m < Q; ++m, ++i) {
            const int sz = i % nz, b = i & 1;
            if (!mbar_wait(&zfull[sz], (i / nz) & 1, a.err)) { ok = false; break; }
            if (i >= 2 && !mbar_wait(&dwfree[b], ((i >> 1) - 1) & 1, a.err)) { ok = false; break; }
            tc_fence_after();
            const uint32_t hs = smem_u32(hb(kt & 1, m)), zs = smem_u32(zb(sz));
            for (int kk = 0; kk < kb; ++kk)
              tc_mma_bf16(tmem + kBwdTmemW + 64 * b, umma_desc_sw128_mn(hs + kk * 2048, tbytes),
                          umma_desc_sw128_mn(zs + kk * 2048, tbytes), idesc_dw, kk > 0 ? 1u : 0u);
            tc_commit(&dwdone[b]);
            tc_commit(&zempty[sz]);
          }
        }
        tc_commit(&hempty[kt & 1]);          // the H tiles are free once these MMAs are
      }
      ok = __all_sync(0xffffffffu, ok);
    }
    if (lane == 0) {
      tc_commit(done);
      mbar_wait(done, 0, a.err);
    }
  } else if constexpr (Q == 1) {
    // ---- warps 0-3: thread t owns input feature i0 + t of the current chunk
    const int t = threadIdx.x;
    const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * warp) << 16);
    int i = 0;
    bool ok = true;
    for (int k = 0; ok; ++k) {
      const int it = take(k);
      if (it < 0) break;
      int tile, c_lo, c_hi;
      decode(it, tile, c_lo, c_hi);
      for (int c = c_lo; c < c_hi && ok; ++c, ++i) {
        const int sw = i % nw, b = i & 1;
        if (!wait_warp(&wfull[sw], (i / nw) & 1, a.err)) { ok = false; break; }
        float* w = reinterpret_cast<float*>(wf(sw));
        float wv[64];
#pragma unroll
        for (int o = 0; o < 64; ++o) wv[o] = w[o * 128 + t];
        if (!wait_warp(&dwdone[b], (i >> 1) & 1, a.err)) { ok = false; break; }
        tc_fence_after();
        // the updated column: w - lr * dW, IEEE multiply then subtract
#pragma unroll
        for (int qb = 0; qb < 4; ++qb) {
          float d[16];
          tmem_ld16(tbase + kBwdTmemW + 64 * b + 16 * qb, d);
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 16; ++q) wv[16 * qb + q] = __fsub_rn(wv[16 * qb + q], __fmul_rn(a.lr, d[q]));
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&dwfree[b]);
#pragma unroll
        for (int o = 0; o < 64; ++o) w[o * 128 + t] = wv[o];
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&upd[sw]);
      }
    }
  } else {
    // ---- warps 0-3 and 8-11: thread (warp % 4, lane) owns input feature i0 + t of the
    // chunk, warps 0-3 its outputs 0-31, warps 8-11 its outputs 32-63
    const int t = 32 * (warp & 3) + lane, o0 = warp >= 8 ? 32 : 0;
    const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
    int i = 0;
    bool ok = true;
    float s0[32], s1[32];                    // partial sums of the pair tree
    for (int k = 0; ok; ++k) {
      const int it = take(k);
      if (it < 0) break;
      int tile, c_lo, c_hi;
      decode(it, tile, c_lo, c_hi);
      for (int c = c_lo; c < c_hi && ok; ++c) {
        for (int m = 0; m < Q; ++m, ++i) {
          const int sw = i % nw, b = i & 1;
          if (!wait_warp(&wfull[sw], (i / nw) & 1, a.err)) { ok = false; break; }
          float* w = reinterpret_cast<float*>(wf(sw)) + o0 * 128;
          if (!wait_warp(&dwdone[b], (i >> 1) & 1, a.err)) { ok = false; break; }
          tc_fence_after();
          // learner m's updated column, w - lr * dW (IEEE multiply then subtract), goes
          // into pair partial m / 2 of the tree (s0 or s1): the first of a pair starts
          // it, the second is added to it
          const bool second = (m & 1) != 0, upper = Q == 4 && m >= 2;
#pragma unroll
          for (int qb = 0; qb < 2; ++qb) {
            float d[16];
            tmem_ld16(tbase + kBwdTmemW + 64 * b + o0 + 16 * qb, d);
            float v[16];
#pragma unroll
            for (int q = 0; q < 16; ++q) v[q] = w[(16 * qb + q) * 128 + t];
            tmem_ld_wait();
#pragma unroll
            for (int q = 0; q < 16; ++q) {
              const int o = 16 * qb + q;
              const float u = __fsub_rn(v[q], __fmul_rn(a.lr, d[q]));
              if (upper)
                s1[o] = second ? __fadd_rn(s1[o], u) : u;
              else
                s0[o] = second ? __fadd_rn(s0[o], u) : u;
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&dwfree[b]);
          if (m + 1 == Q) {
            // the group sum (w0 + w1) or ((w0 + w1) + (w2 + w3)) replaces the last slot
#pragma unroll
            for (int o = 0; o < 32; ++o) w[o * 128 + t] = Q == 4 ? __fadd_rn(s0[o], s1[o]) : s0[o];
            fence_proxy_async_smem();
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(&upd[sw]);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kBwdTmemCols);
  }
  if (threadIdx.x == 0) {
    // the last CTA out resets the counters for the next launch (every claim of every
    // CTA precedes that CTA's increment here)
    __threadfence();
    if (atomicAdd(a.dyn + 1, 1) == static_cast<int>(gridDim.x) - 1) {
      a.dyn[0] = 0;
      a.dyn[1] = 0;
    }
  }
}

// ------------------------------------------------------------------ update + next forward
// The first layer's input is the data, so the forward of the NEXT step's first layer,
// Z_1' = X' W_1'^T (X' = the next batch, W_1' = W_1 after this step's update), can be
// computed by the kernel that produces W_1': this step's first-layer backward.  Then
// W_1 is read once per step instead of twice (update + next forward: 8 bytes per
// weight instead of 12).  The kernel keeps the forward's work items and arithmetic
// exactly (tile = learner j x 128 outputs, chunk = 64 inputs; the same dynamic items
// and tail pieces, or cluster split-K with the same split; the same 4 MMAs per chunk,
// the same every-kSegChunks promotion from the item's first chunk, the same piece
// order), so Z_1' is bit-identical to what k_tc_forward computes from the stored W_1'.
// Per chunk:
//   dW[o][i]  = sum_b dZ_1[b][o] X[b][i]      M = 128 outputs, N = 64 inputs, K = Bn
//                                             (dZ tile and X tile both MN-major)
//   W[o][i]  -= lr dW[o][i]                   fp32, in the shared-memory W tile, which is
//                                             then TMA-stored back
//   Z'^T     += W'_q X'^T                      A = W' rounded to bf16, written to TMEM by
//                                             the thread that owns output row o
// and the tile epilogue writes H_1' = relu(Z' + b_1) (b_1 already updated by the layer
// above).  Warps 0-7 own the accumulator rows as in the forward (row 32*(w%4) + lane,
// input half w/4) and do the update, the bf16 conversion and the drains; warp 8 claims
// the work items and loads W tiles, warp 9 issues the MMAs (the dW MMAs of chunk i
// before the forward MMAs of chunk i-1, so the update of one chunk overlaps the dW of
// the next), warp 10 loads the batch tiles (X and X' rows of the chunk), warp 11
// stores updated W tiles and frees their slots, warp 12 loads the dZ tile of each
// item (two buffers when shared memory allows, so the next item's is loaded ahead).
constexpr int kUfConv = 256;
constexpr int kUfThreads = kUfConv + 160;
// TMEM columns: Z'^T accumulators at 0 and 64, bf16 A tiles at 128 and 160, dW
// accumulators at 256 and 320.
constexpr uint32_t kUfTmemCols = 512, kUfTmemA = 128, kUfTmemDW = 256;

// Layout: W ring | dZ tiles ([Bn][128] bf16, two boxes each) | batch ring (X box, X'
// box per chunk) | barriers.
// nz: dZ tile buffers, two in dynamic mode when shared memory allows (the next item's
// tile loads while this one's is in use), one in cluster mode (one item per CTA).
// (64-row batches: 4 weight slots, so that the batch ring holds 5 chunks instead of 3:
// 3072-2048-2048-10 update+forward 542 -> 535 us; a 4-slot weight ring in the backward,
// for an 8-deep dZ ring, measured slower)
__host__ __device__ constexpr int uf_wring(int Bn) { return Bn > 48 ? 4 : 5; }
__host__ __device__ constexpr int uf_zbufs(int Bn, bool dyn) { return dyn && Bn <= 32 ? 2 : 1; }
__host__ __device__ constexpr int uf_z_off(int Bn) { return uf_wring(Bn) * kFwdWf32; }
__host__ __device__ constexpr int uf_h_off(int Bn, int nz) { return uf_z_off(Bn) + nz * 2 * Bn * 128; }
__host__ __device__ constexpr int uf_hring(int Bn, int nz) {
  return (kFwdSmemMax - 1024 - kBarBytes - uf_h_off(Bn, nz)) / (2 * Bn * 128) < kFwdHRingMax
             ? (kFwdSmemMax - 1024 - kBarBytes - uf_h_off(Bn, nz)) / (2 * Bn * 128)
             : kFwdHRingMax;
}
__host__ __device__ constexpr int uf_bar_off(int Bn, int nz) {
  return uf_h_off(Bn, nz) + uf_hring(Bn, nz) * 2 * Bn * 128;
}
__host__ __device__ constexpr int uf_smem(int Bn, int nz) { return uf_bar_off(Bn, nz) + kBarBytes + 1024; }
// (the cluster split-K partial [128][Bn] fp32 is staged in the batch ring: hring >= 2)
static_assert(uf_hring(64, 1) >= 5 && uf_hring(48, 1) >= 4 && uf_hring(32, 1) >= 7 &&
                  uf_hring(32, 2) >= 6 && uf_hring(16, 2) == 8 && uf_smem(64, 1) <= kFwdSmemMax &&
                  uf_smem(48, 1) <= kFwdSmemMax && uf_smem(32, 2) <= kFwdSmemMax &&
                  uf_smem(16, 2) <= kFwdSmemMax,
              "update+forward shared-memory plan");

template <bool kDyn>
__global__ void __launch_bounds__(kUfThreads, 1)
    k_tc_update_forward(const __grid_constant__ CUtensorMap tm_wl, const __grid_constant__ CUtensorMap tm_ws,
                        const __grid_constant__ CUtensorMap tm_hc, const __grid_constant__ CUtensorMap tm_hn,
                        const __grid_constant__ CUtensorMap tm_dz, const TcFwdArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = blockIdx.x;
  const int nk = (a.in + 63) / 64;
  constexpr bool dyn = kDyn;
  const int cq = kDyn ? 1 : a.cq, part = g % cq;
  const int n_items = a.n_whole + (a.n_tiles - a.n_whole) * a.np_tail;
  const int nz = uf_zbufs(a.Bn, dyn), nw = uf_wring(a.Bn), nh = uf_hring(a.Bn, nz);
  const int tbytes = a.Bn * 128;                            // one [Bn][64] bf16 box
  uint8_t* z_base = smem + uf_z_off(a.Bn);
  uint8_t* h_base = smem + uf_h_off(a.Bn, nz);
  uint64_t* wfull = reinterpret_cast<uint64_t*>(smem + uf_bar_off(a.Bn, nz));
  uint64_t* wempty = wfull + kFwdWRingMax;   // W tile stored back (the TMA has read it)
  uint64_t* upd = wempty + kFwdWRingMax;     // W tile updated in shared memory
  uint64_t* hfull = upd + kFwdWRingMax;
  uint64_t* hempty = hfull + kFwdHRingMax;   // X and X' boxes consumed by both MMAs
  uint64_t* zfull = hempty + kFwdHRingMax;   // [2]
  uint64_t* zempty = zfull + 2;              // [2] dZ tile consumed by the item's dW MMAs
  uint64_t* dwdone = zempty + 2;             // [2] dW of the chunk complete
  uint64_t* dwfree = dwdone + 2;             // [2] dW read by the update
  uint64_t* conv = dwfree + 2;               // [2] A tile written to TMEM
  uint64_t* afree = conv + 2;                // [2] A tile consumed by the forward MMA
  uint64_t* accf = afree + 2;                // [2] accumulator segment complete
  uint64_t* accr = accf + 2;                 // [2] accumulator segment drained
  uint64_t* gbar = accr + 2;
  uint64_t* done = gbar + 1;
  ItemQueue queue{done + 1, done + 1 + kQueue, nullptr};
  queue.items = reinterpret_cast<int*>(done + 1 + 2 * kQueue);
  int* last_flag = queue.items + kQueue;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(last_flag + 1);
  auto wf = [&](int s) { return smem + s * kFwdWf32; };
  auto zb = [&](int s) { return z_base + s * 2 * tbytes; };
  auto hb = [&](int s) { return h_base + s * 2 * tbytes; };
  const FwdItem cl_item{g / cq, part * nk / cq, (part + 1) * nk / cq, 0, 1};
  constexpr int kConsumers = 4 + kUfConv / 32;   // MMA, batch, store, dZ and converter warps

  if (threadIdx.x == 0) {
    for (int s = 0; s < kFwdWRingMax; ++s) {
      mbar_init(&wfull[s], 1);
      mbar_init(&wempty[s], 1);
      mbar_init(&upd[s], kUfConv / 32);
    }
    for (int s = 0; s < kFwdHRingMax; ++s) {
      mbar_init(&hfull[s], 1);
      mbar_init(&hempty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&zfull[b], 1);
      mbar_init(&zempty[b], 1);
      mbar_init(&dwdone[b], 1);
      mbar_init(&dwfree[b], kUfConv / 32);
      mbar_init(&conv[b], kUfConv / 32);
      mbar_init(&afree[b], 1);
      mbar_init(&accf[b], 1);
      mbar_init(&accr[b], kUfConv);
    }
    if (dyn)
      for (int q = 0; q < kQueue; ++q) {
        mbar_init(&queue.full[q], 1);
        mbar_init(&queue.empty[q], kConsumers);
      }
    mbar_init(gbar, kUfConv);
    mbar_init(done, 1);
    fence_barrier_init();
  }
  if (warp == 9) {
    tmem_alloc(tmem_slot, kUfTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  grid_dep_wait();                       // dZ_1 and b_1 of the layer above are visible

  auto next_item = [&](int k, FwdItem& f) -> bool {
    if (!dyn) {
      f = cl_item;
      return k == 0;
    }
    const int it = queue.take(k, lane, a.err);
    if (it < 0) return false;
    f = uf_item(a, nk, it);
    return true;
  };
  // (the batch and dZ tiles are re-read for every output tile: kept in L2)
  const uint64_t keep = l2_keep_policy();

  if (warp == 8) {
    if (lane == 0) {
      // claim (dynamic), announce, and stream the weight tiles
      tma_prefetch_desc(&tm_wl);
      const uint64_t stream = l2_weight_policy(a.w_stream != 0, a.w_div > 1);
      int i = 0, issued = 0;
      bool ok = true;
      int next = dyn ? atomicAdd(a.dyn, 1) : 0;
      for (int k = 0; ok; ++k) {
        FwdItem f;
        if (dyn) {
          const int it = next < n_items ? next : -1;
          if (!queue.put(k, it, a.err) || it < 0) break;
          next = atomicAdd(a.dyn, 1);           // the next claim, hidden behind these loads
          f = uf_item(a, nk, it);
        } else {
          if (k > 0) break;
          f = cl_item;
        }
        const int j = f.tau / a.o_tiles, ot = f.tau - j * a.o_tiles, jw = j / a.w_div;
        for (int c = f.c_lo; c < f.c_hi; ++c, ++i) {
          const int s = i % nw;
          if (i >= nw && !mbar_wait(&wempty[s], ((i / nw) - 1) & 1, a.err)) { ok = false; break; }
          mbar_arrive_expect_tx(&wfull[s], kFwdWf32);
          tma_load_3d_hint(wf(s), &tm_wl, &wfull[s], c * 64, ot * 128, jw, stream);
          tma_load_3d_hint(wf(s) + kFwdWBox, &tm_wl, &wfull[s], c * 64 + 32, ot * 128, jw, stream);
          issued = i + 1;
        }
      }
      for (int u = issued - nw > 0 ? issued - nw : 0; u < issued; ++u)
        mbar_wait(&wfull[u % nw], (u / nw) & 1, a.err);
    }
    if (cq > 1) {
      cluster_sync_all();
      cluster_sync_all();
    }
  } else if (warp == 10) {
    // the X and X' boxes of each chunk
    if (lane == 0) {
      tma_prefetch_desc(&tm_hc);
      tma_prefetch_desc(&tm_hn);
    }
    int i = 0, issued = 0;
    bool ok = true;
    FwdItem f;
    for (int k = 0; ok && next_item(k, f); ++k) {
      if (lane == 0) {
        const int j = f.tau / a.o_tiles;
        for (int c = f.c_lo; c < f.c_hi; ++c, ++i) {
          const int s = i % nh;
          if (i >= nh && !mbar_wait(&hempty[s], ((i / nh) - 1) & 1, a.err)) { ok = false; break; }
          mbar_arrive_expect_tx(&hfull[s], 2 * tbytes);
          tma_load_3d_hint(hb(s), &tm_hc, &hfull[s], c * 64, a.hc_row0, j, keep);
          tma_load_3d_hint(hb(s) + tbytes, &tm_hn, &hfull[s], c * 64, a.x_row0, j, keep);
          issued = i + 1;
        }
      }
      ok = __all_sync(0xffffffffu, ok);
    }
    if (lane == 0)
      for (int u = issued - nh > 0 ? issued - nh : 0; u < issued; ++u)
        mbar_wait(&hfull[u % nh], (u / nh) & 1, a.err);
    if (cq > 1) {
      cluster_sync_all();
      cluster_sync_all();
    }
  } else if (warp == 12) {
    // the dZ tile (128 outputs x Bn) of each item
    if (lane == 0) tma_prefetch_desc(&tm_dz);
    int zissued = 0;
    bool ok = true;
    FwdItem f;
    for (int v = 0; ok && next_item(v, f); ++v) {
      if (lane == 0) {
        const int j = f.tau / a.o_tiles, ot = f.tau - j * a.o_tiles;
        const int zs = v % nz;
        if (v >= nz && !mbar_wait(&zempty[zs], ((v / nz) - 1) & 1, a.err)) {
          ok = false;
        } else {
          mbar_arrive_expect_tx(&zfull[zs], 2 * tbytes);
          tma_load_3d_hint(zb(zs), &tm_dz, &zfull[zs], ot * 128, 0, j, keep);
          tma_load_3d_hint(zb(zs) + tbytes, &tm_dz, &zfull[zs], ot * 128 + 64, 0, j, keep);
          zissued = v + 1;
        }
      }
      ok = __all_sync(0xffffffffu, ok);
    }
    if (lane == 0)
      for (int v = zissued - nz > 0 ? zissued - nz : 0; v < zissued; ++v)
        mbar_wait(&zfull[v % nz], (v / nz) & 1, a.err);
    if (cq > 1) {
      cluster_sync_all();
      cluster_sync_all();
    }
  } else if (warp == 11) {
    // Store each updated W tile; its slot is released once the TMA has read it.  In
    // cluster mode (a short layer), and when the tiles come from the cluster means (the
    // first step of a block, which the SMs' chunk rate bounds, not DRAM), each slot is
    // released as soon as its own store has been read; otherwise one store behind, two
    // in flight.
    const uint64_t stream = l2_weight_policy(a.w_stream != 0);
    const bool eager = cq > 1 || a.w_div > 1;
    int i = 0, released = 0;
    bool ok = true;
    FwdItem f;
    for (int k = 0; ok && next_item(k, f); ++k) {
      if (lane == 0) {
        const int j = f.tau / a.o_tiles, ot = f.tau - j * a.o_tiles;
        for (int c = f.c_lo; c < f.c_hi; ++c, ++i) {
          const int s = i % nw;
          if (!mbar_wait(&upd[s], (i / nw) & 1, a.err)) { ok = false; break; }
          tma_store_3d_hint(&tm_ws, wf(s), c * 64, ot * 128, j, stream);
          tma_store_3d_hint(&tm_ws, wf(s) + kFwdWBox, c * 64 + 32, ot * 128, j, stream);
          tma_store_commit();
          if (eager) {
            tma_store_wait_read_all();
            mbar_arrive(&wempty[s]);
            released = i + 1;
          } else if (i > 0) {
            tma_store_wait_read_1();
            mbar_arrive(&wempty[(i - 1) % nw]);
            released = i;
          }
        }
      }
      ok = __all_sync(0xffffffffu, ok);
    }
    if (lane == 0) {
      tma_store_wait_read_all();   // (before the shared memory is released)
      if (i > released) mbar_arrive(&wempty[(i - 1) % nw]);
    }
    if (cq > 1) {
      cluster_sync_all();
      cluster_sync_all();
    }
  } else if (warp == 9) {
    const uint32_t idesc_dw = umma_idesc_bf16(128, 64) | (1u << 15) | (1u << 16);
    const uint32_t idesc_fw = umma_idesc_bf16(128, a.Bn);
    const int kb = a.Bn / 16;
    // Forward MMAs of chunk k into accumulator segment qq (first/last: of the segment).
    auto fwd = [&](int k, bool first, bool last, int qq) -> bool {
      const int ab = qq & 1, bb = k & 1, sh = k % nh;
      if (first && qq >= 2 && !mbar_wait(&accr[ab], ((qq >> 1) - 1) & 1, a.err)) return false;
      if (!mbar_wait(&conv[bb], (k >> 1) & 1, a.err)) return false;
      tc_fence_after();
      const uint32_t at = tmem + kUfTmemA + 32 * bb;
      const uint64_t bd = umma_desc_sw128(smem_u32(hb(sh) + tbytes));
      const uint32_t d = tmem + 64 * ab;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        tc_mma_bf16_ta(d, at + 8 * kk, bd + 2 * kk, idesc_fw, (!first || kk > 0) ? 1u : 0u);
      tc_commit(&hempty[sh]);
      tc_commit(&afree[bb]);
      if (last) tc_commit(&accf[ab]);
      return true;
    };
    int i = 0, q = -1;
    int pend = -1, pend_q = 0;
    bool pend_first = false, pend_last = false, ok = true;
    FwdItem f;
    for (int v = 0; ok && next_item(v, f); ++v) {
      if (lane == 0) {
        const int zs = v % nz;
        // The pending forward (last chunk of the previous item) goes first if this
        // item's dZ tile has not arrived yet, so that the converters can close that item.
        if (pend >= 0 && !mbar_test(&zfull[zs], (v / nz) & 1)) {
          if (!fwd(pend, pend_first, pend_last, pend_q)) ok = false;
          pend = -1;
        }
        if (ok && !mbar_wait(&zfull[zs], (v / nz) & 1, a.err)) ok = false;
        const uint32_t zsa = smem_u32(zb(zs));
        for (int c = f.c_lo, p = 0; ok && c < f.c_hi; ++c, ++p, ++i) {
          const bool tlast = c == f.c_hi - 1;
          const bool first = p % kSegChunks == 0, last = tlast || p % kSegChunks == kSegChunks - 1;
          if (first) ++q;
          const int sh = i % nh, bb = i & 1;
          if (!mbar_wait(&hfull[sh], (i / nh) & 1, a.err)) { ok = false; break; }
          if (i >= 2 && !mbar_wait(&dwfree[bb], ((i >> 1) - 1) & 1, a.err)) { ok = false; break; }
          tc_fence_after();
          const uint32_t hs = smem_u32(hb(sh));
          for (int kk = 0; kk < kb; ++kk)
            tc_mma_bf16(tmem + kUfTmemDW + 64 * bb, umma_desc_sw128_mn(zsa + kk * 2048, tbytes),
                        umma_desc_sw128_mn(hs + kk * 2048, tbytes), idesc_dw, kk > 0 ? 1u : 0u);
          tc_commit(&dwdone[bb]);
          if (tlast) tc_commit(&zempty[zs]);
          if (pend >= 0 && !fwd(pend, pend_first, pend_last, pend_q)) { ok = false; break; }
          pend = i;
          pend_first = first;
          pend_last = last;
          pend_q = q;
        }
      }
      ok = __all_sync(0xffffffffu, ok);
    }
    if (lane == 0) {
      if (ok && pend >= 0) fwd(pend, pend_first, pend_last, pend_q);
      tc_commit(done);
      mbar_wait(done, 0, a.err);   // no MMA may be in flight at teardown
    }
    if (cq > 1) {
      cluster_sync_all();
      cluster_sync_all();
    }
  } else {
    // ---- warps 0-7: the update, the bf16 A tile, the drains and the tile epilogues
    const int t = threadIdx.x;
    const int r = t & 127, gr = t >> 7;                    // accumulator row, column group
    const int row = 32 * (warp & 3) + lane, half = warp >> 2;   // (row == r)
    const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
    GroupSync gsync{gbar, 0, a.err};
    float acc[32];
#pragma unroll
    for (int q = 0; q < 32; ++q) acc[q] = 0.f;
    int qc = -1, drained = 0;
    auto drain = [&]() -> bool {
      const int ab = drained & 1;
      if (!wait_warp(&accf[ab], (drained >> 1) & 1, a.err)) return false;
      tc_fence_after();
#pragma unroll
      for (int m = 0; m < 2; ++m) {
        const int cb = (2 * m + gr) * 16;
        if (cb < a.Bn) {
          float v[16];
          tmem_ld16(tbase + 64 * ab + cb, v);
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 16; ++q) acc[16 * m + q] = __fadd_rn(acc[16 * m + q], v[q]);
        }
      }
      tc_fence_before();
      mbar_arrive(&accr[ab]);
      ++drained;
      return true;
    };
    // As the forward's hidden-layer epilogue: H_1'[j][b][o] = relu(Z' + b_1).  The
    // cluster build loads the bias of its one tile up front (cl_bias); the dynamic build,
    // short of registers, at the epilogue.
    const int cl_o = (cl_item.tau % a.o_tiles) * 128 + r;
    const float cl_bias =
        !kDyn && cl_o < a.out
            ? a.bias[static_cast<int64_t>(cl_item.tau / a.o_tiles / a.b_div) * a.ld + cl_o]
            : 0.f;
    auto epilogue = [&](int tau) {
      const int j = tau / a.o_tiles, ot = tau - j * a.o_tiles;
      const int o = ot * 128 + r;
      if (o < a.out) {
        const float bias = kDyn ? a.bias[static_cast<int64_t>(j / a.b_div) * a.ld + o] : cl_bias;
#pragma unroll
        for (int m = 0; m < 2; ++m) {
          const int cb = (2 * m + gr) * 16;
          if (cb >= a.Bn) break;
#pragma unroll
          for (int q = 0; q < 16; ++q)
            if (cb + q < a.B)
              a.h_out[(static_cast<int64_t>(j) * a.Bn + cb + q) * a.pitch_out + o] =
                  __float2bfloat16_rn(fmaxf(__fadd_rn(acc[16 * m + q], bias), 0.f));
        }
      }
    };
    bool ok = true, have_ep = false;   // have_ep: cluster split-K, this CTA's part is done
    int i = 0;
    FwdItem f;
    for (int k = 0; ok && next_item(k, f); ++k) {
      for (int c = f.c_lo, p = 0; c < f.c_hi && ok; ++c, ++p, ++i) {
        const bool tlast = c == f.c_hi - 1;
        const int sw = i % nw, bb = i & 1;
        if (!wait_warp(&wfull[sw], (i / nw) & 1, a.err)) { ok = false; break; }
        if (!wait_warp(&dwdone[bb], (i >> 1) & 1, a.err)) { ok = false; break; }
        tc_fence_after();
        float d[32];
        tmem_ld16(tbase + kUfTmemDW + 64 * bb + 32 * half, d);
        tmem_ld16(tbase + kUfTmemDW + 64 * bb + 32 * half + 16, d + 16);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&dwfree[bb]);
        // W[o][32*half + 4q ..] sits in 16-byte chunk q ^ (o % 8) of row o of box `half`
        uint8_t* src = wf(sw) + half * kFwdWBox + row * 128;
        uint32_t pk[16];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          float4* pw = reinterpret_cast<float4*>(src + ((q ^ (row & 7)) << 4));
          float4 x = *pw;
          x.x = __fsub_rn(x.x, __fmul_rn(a.lr, d[4 * q]));
          x.y = __fsub_rn(x.y, __fmul_rn(a.lr, d[4 * q + 1]));
          x.z = __fsub_rn(x.z, __fmul_rn(a.lr, d[4 * q + 2]));
          x.w = __fsub_rn(x.w, __fmul_rn(a.lr, d[4 * q + 3]));
          *pw = x;
          pk[2 * q] = pack_bf16x2(x.x, x.y);
          pk[2 * q + 1] = pack_bf16x2(x.z, x.w);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&upd[sw]);
        if (i >= 2 && !wait_warp(&afree[bb], ((i >> 1) - 1) & 1, a.err)) { ok = false; break; }
        tc_fence_after();
        tmem_st16(tbase + kUfTmemA + 32 * bb + 16 * half, pk);
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&conv[bb]);
        if (p % kSegChunks == 0) ++qc;
        if (tlast) {
          while (ok && drained <= qc)
            if (!drain()) ok = false;
          if (!ok) break;
          if (!dyn) {
            have_ep = true;
            if (part != 0) {
              // the batch ring is idle once the last segment is drained
              float* red = reinterpret_cast<float*>(h_base) + r * a.Bn;
#pragma unroll
              for (int m = 0; m < 2; ++m) {
                const int cb = (2 * m + gr) * 16;
                if (cb < a.Bn) {
#pragma unroll
                  for (int q = 0; q < 16; q += 4)
                    *reinterpret_cast<float4*>(red + cb + q) =
                        make_float4(acc[16 * m + q], acc[16 * m + q + 1], acc[16 * m + q + 2],
                                    acc[16 * m + q + 3]);
                }
              }
            }
          } else {
            const bool fin = f.np == 1 || piece_end(a, f, t, r, gr, acc, gsync, last_flag, ok);
            if (ok && fin) epilogue(f.tau);
#pragma unroll
            for (int q = 0; q < 32; ++q) acc[q] = 0.f;
            ok = __all_sync(0xffffffffu, ok);
          }
        } else if (p % kSegChunks == kSegChunks - 1 && qc >= 1 && drained < qc) {
          if (!drain()) ok = false;
        }
      }
    }
    if (cq > 1) {
      cluster_sync_all();
      if (part == 0 && __all_sync(0xffffffffu, ok && have_ep)) {
        for (int rk = 1; rk < cq; ++rk) {
          const float* red = reinterpret_cast<const float*>(h_base) + r * a.Bn;
#pragma unroll
          for (int m = 0; m < 2; ++m) {
            const int cb = (2 * m + gr) * 16;
            if (cb < a.Bn) {
#pragma unroll
              for (int q = 0; q < 16; q += 4) {
                const float4 v = ld_cluster_f4(red + cb + q, rk);
                acc[16 * m + q] = __fadd_rn(acc[16 * m + q], v.x);
                acc[16 * m + q + 1] = __fadd_rn(acc[16 * m + q + 1], v.y);
                acc[16 * m + q + 2] = __fadd_rn(acc[16 * m + q + 2], v.z);
                acc[16 * m + q + 3] = __fadd_rn(acc[16 * m + q + 3], v.w);
              }
            }
          }
        }
        epilogue(cl_item.tau);
      }
      cluster_sync_all();
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kUfTmemCols);
  }
  if (dyn && threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(a.dyn + 1, 1) == static_cast<int>(gridDim.x) - 1) {
      a.dyn[0] = 0;
      a.dyn[1] = 0;
    }
  }
}

// ------------------------------------------------------------------ gather
// H_0[j][b][:] = X[j][(row0 + b) mod N][:] for b < B, one CTA per (64-feature slice,
// learner); rows b >= B stay zero.
__global__ void __launch_bounds__(256) k_gather_bf16(const __nv_bfloat16* __restrict__ X,
                                                    int64_t N, int d0, int B, int Bn,
                                                    int pitch0, int64_t row0,
                                                    __nv_bfloat16* __restrict__ H0) {
  grid_dep_wait();
  const int j = blockIdx.y, k0 = blockIdx.x * 64;
  const int nvec = B * 8;                       // 16-byte vectors in the [B][64] slice
  for (int idx = threadIdx.x; idx < nvec; idx += blockDim.x) {
    const int b = idx >> 3, v = idx & 7;
    const int k = k0 + v * 8;
    if (k < d0) {
      const int64_t row = (row0 + b) % N;
      *reinterpret_cast<uint4*>(H0 + (static_cast<int64_t>(j) * Bn + b) * pitch0 + k) =
          *reinterpret_cast<const uint4*>(X + (static_cast<int64_t>(j) * N + row) * d0 + k);
    }
  }
}

// ------------------------------------------------------------------ cross-entropy
// Softmax cross-entropy gradient when the classes span several output tiles.
// Grid (P, class slices of 1024).  Every CTA computes the per-sample statistics
// (max, sum of exponentials over all C classes) with one warp per sample, then each
// thread owns one class of its slice: dZ = (p - onehot(y_b)) / B in fp32 for every
// sample, its bf16 copy, and b_L -= lr * sum_b dZ (summed in sample order).  Slice 0
// also writes the learner's mean loss.  (The statistics are a chain of dependent
// loads; a warp per sample keeps that chain to one row.  With 256-thread CTAs, four
// per learner at 1000 classes, each warp walked four rows one after the other: 23.1
// against 18.9 us per launch at B = 32, P = 32.)
constexpr int kXentThreads = 1024;
__global__ void __launch_bounds__(kXentThreads, 1) k_xent_bf16(const float* __restrict__ Z,
                                                              const int32_t* __restrict__ y,
                                                              int64_t N, int64_t row0, int B, int Bn,
                                                              int C, int pitch_c, float lr,
                                                              const float* bias_src,
                                                              int src_div, float* bias_L, int64_t ld,
                                                              __nv_bfloat16* dZ, float* loss) {
  __shared__ float row_max[64], row_sum[64], row_loss[64];
  __shared__ int row_y[64];
  grid_dep_wait();
  const int j = blockIdx.x, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* Zj = Z + static_cast<int64_t>(j) * B * C;
  // (Each lane's classes c = lane, lane + 32, ... in increasing order, eight loads in
  // flight at a time: one load at a time left the kernel waiting on L2 latency, and a
  // lane's whole row in registers at once, 32 loads, measured slower.)
  for (int b = warp; b < B; b += kXentThreads / 32) {
    const float* z = Zj + static_cast<int64_t>(b) * C;
    float m = -INFINITY;
    for (int c0 = 0; c0 < C; c0 += 256) {
      float v[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int c = c0 + lane + 32 * k;
        v[k] = c < C ? z[c] : -INFINITY;
      }
#pragma unroll
      for (int k = 0; k < 8; ++k)
        if (c0 + lane + 32 * k < C) m = fmaxf(m, v[k]);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
    float s = 0.f;
    for (int c0 = 0; c0 < C; c0 += 256) {
      float v[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int c = c0 + lane + 32 * k;
        v[k] = c < C ? z[c] : 0.f;
      }
#pragma unroll
      for (int k = 0; k < 8; ++k)
        if (c0 + lane + 32 * k < C) s += expf(v[k] - m);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) {
      const int yb = y[static_cast<int64_t>(j) * N + (row0 + b) % N];
      row_max[b] = m;
      row_sum[b] = s;
      row_y[b] = yb;
      row_loss[b] = logf(s) + m - z[yb];
    }
  }
  __syncthreads();
  if (blockIdx.y == 0 && threadIdx.x == 0) {
    float l = 0.f;
    for (int b = 0; b < B; ++b) l += row_loss[b];
    loss[j] = l / B;
  }
  const int c = blockIdx.y * kXentThreads + threadIdx.x;
  if (c >= C) return;
  // (bias_src may be bias_L itself: read before the write below)
  const float bv = bias_src[static_cast<int64_t>(j / src_div) * ld + c];
  const float fB = static_cast<float>(B);
  float db = 0.f;
  for (int b0 = 0; b0 < B; b0 += 8) {
    float zv[8];
#pragma unroll
    for (int k = 0; k < 8; ++k)
      zv[k] = b0 + k < B ? Zj[static_cast<int64_t>(b0 + k) * C + c] : 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int b = b0 + k;
      if (b < B) {
        const float p = __fdiv_rn(expf(zv[k] - row_max[b]), row_sum[b]);
        const float g = __fdiv_rn(__fsub_rn(p, row_y[b] == c ? 1.f : 0.f), fB);
        db = __fadd_rn(db, g);
        dZ[(static_cast<int64_t>(j) * Bn + b) * pitch_c + c] = __float2bfloat16_rn(g);
      }
    }
  }
  bias_L[static_cast<int64_t>(j) * ld + c] = __fsub_rn(bv, __fmul_rn(lr, db));
}

}  // namespace

int tc_fwd_smem_bytes() { return kFwdSmemMax; }
int tc_bwd_smem_bytes() { return kBwdSmemMax; }

cudaError_t tc_configure() {
  cudaError_t e = cudaFuncSetAttribute(k_tc_forward<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       kFwdSmemMax);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_tc_forward<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, kFwdSmemMax);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_tc_forward_group, cudaFuncAttributeMaxDynamicSharedMemorySize, kFwdSmemMax);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_tc_update_forward<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           kFwdSmemMax);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_tc_backward<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, kBwdSmemMax);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_tc_backward<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, kBwdSmemMax);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_tc_update<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, kBwdSmemMax);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_tc_update<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, kBwdSmemMax);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_tc_update<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, kBwdSmemMax);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_tc_update_forward<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              kFwdSmemMax);
}

cudaError_t launch_tc_forward(const CUtensorMap& w_fwd, const CUtensorMap& h_in,
                              const TcFwdArgs& a, int P, cudaStream_t s) {
  (void)P;
  // No CTA waits for another (dynamic items; cluster split-K reduces inside a cluster),
  // so an ordinary launch.
  if (a.cq > 1)
    return launch_pdl(k_tc_forward<false>, dim3(a.ctas), dim3(kFwdThreads), fwd_smem(a.mode, a.Bn), s,
                      false, a.cq, w_fwd, h_in, a);
  return launch_pdl(k_tc_forward<true>, dim3(a.ctas), dim3(kFwdThreads), fwd_smem(a.mode, a.Bn), s,
                    false, 1, w_fwd, h_in, a);
}

int tc_forward_group_size(int S, int Bn) {
  for (int G = 128 / Bn; G >= 2; --G)
    if (S % G == 0) return G;
  return 1;
}

cudaError_t launch_tc_forward_group(const CUtensorMap& w_fwd, const CUtensorMap& h_in,
                                    const TcFwdArgs& a, int G, cudaStream_t s) {
  if (G < 2 || G * a.Bn > 128 || a.n_tiles % G != 0 || a.n_whole % (G * a.o_tiles) != 0 ||
      a.mode == kFwdXent)
    return cudaErrorInvalidValue;
  return launch_pdl(k_tc_forward_group, dim3(a.ctas), dim3(kFwdThreads), gf_smem(G * a.Bn), s, false,
                    1, w_fwd, h_in, a, G);
}

cudaError_t launch_tc_backward(const CUtensorMap& w_load, const CUtensorMap& w_store,
                               const CUtensorMap& h_in, const CUtensorMap& dz, const TcBwdArgs& a,
                               int P, cudaStream_t s) {
  (void)P;
  // dynamic work items, no CTA waits for another: an ordinary launch
  if (a.no_update)
    return launch_pdl(k_tc_backward<true>, dim3(a.ctas), dim3(kBxThreads), bwd_smem(a.Bn), s, false, 1,
                      w_load, w_store, h_in, dz, a);
  return launch_pdl(k_tc_backward<false>, dim3(a.ctas), dim3(kBxThreads), bwd_smem(a.Bn), s, false, 1,
                    w_load, w_store, h_in, dz, a);
}

cudaError_t launch_tc_update(const CUtensorMap& w_load, const CUtensorMap& w_store,
                             const CUtensorMap& h_in, const CUtensorMap& dz, const TcBwdArgs& a,
                             int group, cudaStream_t s) {
  // Items of kRun chunks per learner, unless a group of learners then leaves fewer than
  // 4 items per CTA: then kRun / group chunks per learner (the same work per item).
  TcBwdArgs b = a;
  const int nc = (a.out + 63) / 64;
  b.run = kRun;
  if (group > 1 && static_cast<int64_t>(a.n_tiles / group) * ((nc + kRun - 1) / kRun) < 4 * a.ctas)
    b.run = kRun / group > 0 ? kRun / group : 1;
  // no CTA waits on another: an ordinary (programmatically serialised) launch
  if (group == 4 && a.Bn <= 32)
    return launch_pdl(k_tc_update<4>, dim3(a.ctas), dim3(upd_threads(4)), updg_smem(4, a.Bn), s, false, 1,
                      w_load, w_store, h_in, dz, b);
  if (group == 2)
    return launch_pdl(k_tc_update<2>, dim3(a.ctas), dim3(upd_threads(2)), updg_smem(2, a.Bn), s, false, 1,
                      w_load, w_store, h_in, dz, b);
  if (group != 1) return cudaErrorInvalidValue;
  return launch_pdl(k_tc_update<1>, dim3(a.ctas), dim3(upd_threads(1)), upd_smem(a.Bn), s, false, 1,
                    w_load, w_store, h_in, dz, b);
}

int tc_update_max_group(int Bn) { return Bn <= 32 ? 4 : 2; }

cudaError_t launch_tc_update_forward(const CUtensorMap& w_load, const CUtensorMap& w_store,
                                     const CUtensorMap& h_cur, const CUtensorMap& x_next,
                                     const CUtensorMap& dz, const TcFwdArgs& a, cudaStream_t s) {
  // an ordinary launch, as the forward
  if (a.cq > 1)
    return launch_pdl(k_tc_update_forward<false>, dim3(a.ctas), dim3(kUfThreads),
                      uf_smem(a.Bn, uf_zbufs(a.Bn, false)), s, false, a.cq, w_load, w_store, h_cur,
                      x_next, dz, a);
  return launch_pdl(k_tc_update_forward<true>, dim3(a.ctas), dim3(kUfThreads),
                    uf_smem(a.Bn, uf_zbufs(a.Bn, true)), s, false, 1, w_load, w_store, h_cur, x_next,
                    dz, a);
}

cudaError_t launch_gather_bf16(const __nv_bfloat16* X, int64_t N, int d0, int B, int Bn,
                               int pitch0, int64_t row0, int P, __nv_bfloat16* H0, cudaStream_t s) {
  dim3 grid((d0 + 63) / 64, P);
  return launch_pdl(k_gather_bf16, grid, dim3(256), 0, s, false, 1, X, N, d0, B, Bn, pitch0, row0, H0);
}

cudaError_t launch_xent_bf16(const float* Z, const int32_t* y, int64_t N, int64_t row0, int B,
                             int Bn, int C, int pitch_c, float lr, const float* bias_src,
                             int src_div, float* bias_L, int64_t ld, __nv_bfloat16* dZ,
                             float* loss, int P, cudaStream_t s) {
  dim3 grid(P, (C + kXentThreads - 1) / kXentThreads);
  return launch_pdl(k_xent_bf16, grid, dim3(kXentThreads), 0, s, false, 1, Z, y, N, row0, B, Bn, C,
                    pitch_c, lr, bias_src, src_div, bias_L, ld, dZ, loss);
}

}  // namespace ha
