// Internal declarations shared by the C-ABI layer and the kernel translation units.
#pragma once
#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "hier_avg.h"

namespace ha {

// Launch through cudaLaunchKernelEx with programmatic stream serialization (the
// kernel calls grid_dep_wait() before its first global access), optionally
// cooperative (all CTAs resident at once) or as clusters of cluster_x CTAs.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, bool cooperative, unsigned cluster_x, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[3];
  unsigned n = 0;
  attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[n].val.programmaticStreamSerializationAllowed = 1;
  ++n;
  if (cooperative) {
    attr[n].id = cudaLaunchAttributeCooperative;
    attr[n].val.cooperative = 1;
    ++n;
  }
  if (cluster_x > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster_x;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// ----------------------------------------------------------------- averaging
// Means over groups of n consecutive rows of w[P, ld] (n | P), written back to
// every row of the group.  n = 1 is a no-op.
cudaError_t launch_group_mean(float* w, int64_t P, int64_t n, int64_t D, int64_t ld,
                              cudaStream_t s);
// The same means written once per group, to row g of out[P / n, ld] (w unchanged).
cudaError_t launch_group_mean_to(const float* w, int64_t P, int64_t n, int64_t D, int64_t ld,
                                 float* out, cudaStream_t s);
// Rows of w (stride ld) in groups of n consecutive rows: the adjacent-pair tree sum of
// each group divided by div, to row g of out (stride out_ld).  With div = n this is
// launch_group_mean_to; with rows that are sums of the first tree levels (Q learners
// each, n = S / Q, div = S) it finishes a local average from them.
cudaError_t launch_group_sum_mean_to(const float* w, int64_t rows, int64_t n, int64_t D, int64_t ld,
                                     float div, float* out, int64_t out_ld, cudaStream_t s);
// The local average (clusters of S) followed by the global average, in one pass.
cudaError_t launch_local_global_mean(float* w, int64_t P, int64_t S, int64_t D, int64_t ld,
                                     cudaStream_t s);
// The same, with each cluster's sum taken from S / Q rows of src (stride src_ld) that
// hold sums of Q learners in the first levels of its adjacent-pair tree (Q = 1, 2 or 4,
// Q | S); the result goes to all P rows of w (src may point into w).
cudaError_t launch_local_global_from_groups(const float* src, int64_t src_ld, int64_t Q, float* w,
                                            int64_t P, int64_t S, int64_t D, int64_t ld,
                                            cudaStream_t s);

// ----------------------------------------------------------------- bf16 tensor-core step
// Activation buffers of the bf16 path (all zero-initialised once; kernels only
// ever write the valid region, so the padding stays zero):
//   H_l   [P][Bn][pitch(d_l)]  bf16  layer-l input rows (batch-major)
//   dZ_l  [P][Bn][pitch(d_l)]  bf16  gradient w.r.t. the pre-activation of layer l
//   Z_L   [P][B][d_L]          fp32  logits of the last layer
// Bn = B rounded up to 16 (the MMA N extent, B <= 64), pitch(d) = d rounded up to
// 64.  The backward reads H and dZ as stored (MN-major operands), so no transposed
// copies exist.
// Small last layer (<= 16 classes) on CUDA cores: one kernel, a thread-block cluster
// of feature slices per learner (forward, softmax-CE and backward).
struct HeadArgs {
  int C, in, B, Bn, pitch_in;
  int64_t ld, N;
  int64_t row0;               // first row of this step's batch in each learner's data (< N)
  float lr;
  float* W;                   // learner 0's W_L [C][in] (fp32 master), written
  float* bias;                // learner 0's b_L, written
  // Parameters are read from row j / src_div of these (learner j; the same as W, bias,
  // bias_prev with src_div = 1, or the cluster means right after a compact average).
  const float* W_src;
  const float* bias_src;
  const float* bias_prev_src;
  int src_div;
  const __nv_bfloat16* H;     // H_{L-1} [P][Bn][pitch_in], or X [P][N][in] when x_rows
  int x_rows;
  const int32_t* y;
  int has_dx;                 // write dZ_{L-1} and update b_{L-1}
  float* bias_prev;
  __nv_bfloat16* dz_prev;     // [P][Bn][pitch_in]
  float* loss;                // [P]
};
struct TcFwdArgs {
  int in, out, B, Bn;
  int64_t ld;                 // parameter row length (floats)
  const float* bias;          // b_l read for learner j at row j / b_div (+ row * ld)
  int b_div;
  int w_div;                  // learner j's W is row j / w_div of the W map it is given
  float* bias_out;            // mode 2: b_L after its update, learner j at + j * ld
  int mode;                   // 0 hidden (ReLU -> H), 1 logits -> z_out, 2 fused softmax-CE
  __nv_bfloat16* h_out;       // mode 0: H_{l+1} [P][Bn][pitch_out]
  int pitch_out;              // mode 0: H pitch; mode 2: dZ_L pitch
  float* z_out;               // mode 1: Z_L [P][B][out]
  // Schedule over n_tiles = P x o_tiles tiles (learner x 128 outputs), each reduced over
  // ceil(in/64) chunks.  cq > 1: cluster split-K, ctas = n_tiles * cq.  Otherwise
  // dynamic: `ctas` CTAs claim work items from dyn[0] (dyn[1] counts the CTAs done;
  // both zero on entry, reset on exit).  Tiles [0, n_whole) are one item each; tiles
  // [n_whole, n_tiles) are split into np_tail pieces of piece_chunks chunks.  Piece p
  // of tail tile tt = tau - n_whole writes its partial to part[((tt * np_tail + p) *
  // 128 + row) * Bn + col] and counts itself in counters[tt]; the last one adds the
  // tile's partials in piece order, runs the epilogue and resets counters[tt] to 0.
  int ctas, n_tiles, o_tiles;
  int cq;
  int n_whole, np_tail, piece_chunks;
  float* part;
  int* counters;
  int* dyn;
  // first layer: the batch tile is read straight from X (rows x_row0 .. of learner j)
  int x_direct, x_row0;
  int hc_row0;                // update+forward: rows of this step's batch in its map
  int w_stream;               // load W with the L2 evict-first policy
  // mode 2: labels and outputs of the fused cross-entropy
  const int32_t* y;
  int64_t N, row0;            // labels: rows row0 + b (mod N)
  float lr;
  __nv_bfloat16* dz_out;      // dZ_L [P][Bn][pitch_out]
  float* loss;                // [P]
  int* err;
};
struct TcBwdArgs {
  int in, out, B, Bn;
  int64_t ld;
  float lr;
  int has_dx;                 // compute dZ_{l-1} (every layer but the first)
  int no_update;              // k_tc_backward: dZ_{l-1} and b_{l-1} only; W_l is neither
                              // updated nor stored (a grouped update follows)
  float* bias_prev;           // learner 0's b_{l-1}, written (row j)
  const float* bias_prev_src; // b_{l-1} read for learner j at row j / src_div
  int src_div;                // learner j's W (and b_{l-1}) read from row j / src_div of
                              // the load map (and bias_prev_src)
  __nv_bfloat16* dz_prev;     // dZ_{l-1} [P][Bn][pitch_in]
  int pitch_in;
  int h_row0;                 // first batch row of H_{l-1} in its tensor map (X rows for l = 0)
  int w_stream;               // load and store W with the L2 evict-first policy
  // n_tiles = P x s_tiles tiles (learner x 128 inputs) of ceil(out/64) chunks each,
  // claimed dynamically by `ctas` CTAs from dyn[0] (dyn[1] counts the CTAs done; both
  // zero on entry, reset on exit).  k_tc_backward: tiles [0, n_whole) whole, tiles
  // [n_whole, n_tiles) in np_tail pieces of piece_chunks chunks, dX partials and
  // counters as the forward's.  k_tc_update: runs of up to `run` chunks (set by its
  // launcher).
  int ctas, n_tiles, s_tiles;
  int run;
  int n_whole, np_tail, piece_chunks;
  float* part;
  int* counters;
  int* dyn;
  int* err;
};
int tc_fwd_smem_bytes();
int tc_bwd_smem_bytes();
cudaError_t tc_configure();   // raises the dynamic shared-memory limits once
cudaError_t launch_tc_forward(const CUtensorMap& w_fwd, const CUtensorMap& h_in,
                              const TcFwdArgs& a, int P, cudaStream_t s);
// The forward of groups of G learners that share their weights (the first step after
// a compact local average, a.w_div = a.b_div = S, G | S): one product of each weight
// tile with the G stacked batch tiles, bit-identical to launch_tc_forward.  Dynamic
// schedule only (a.cq == 1), modes 0 and 1; a.n_whole must be a multiple of
// G * a.o_tiles; a.ctas CTAs claim (n_whole + (n_tiles - n_whole) * np_tail) / G items.
cudaError_t launch_tc_forward_group(const CUtensorMap& w_fwd, const CUtensorMap& h_in,
                                    const TcFwdArgs& a, int G, cudaStream_t s);
// The largest G <= 128 / Bn dividing S (1: none above 1).
int tc_forward_group_size(int S, int Bn);
// W is loaded through w_load (row j / a.src_div) and stored through w_store (row j).
cudaError_t launch_tc_backward(const CUtensorMap& w_load, const CUtensorMap& w_store,
                               const CUtensorMap& h_in, const CUtensorMap& dz, const TcBwdArgs& a,
                               int P, cudaStream_t s);
// The first layer's backward (no dX): dW, update and store only, units claimed
// dynamically (a.dyn zero on entry; reset by the kernel on exit).  a.n_tiles = P *
// s_tiles.  group = 1: every learner's W is stored through w_store (row j).  group = 2
// or 4 (at most tc_update_max_group(Bn)): learners g*group .. g*group+group-1 are
// updated together and only their adjacent-pair tree sum is stored, to row g of w_store.
cudaError_t launch_tc_update(const CUtensorMap& w_load, const CUtensorMap& w_store,
                             const CUtensorMap& h_in, const CUtensorMap& dz, const TcBwdArgs& a,
                             int group, cudaStream_t s);
int tc_update_max_group(int Bn);
// The first layer's backward (dW, update, store) fused with the next step's first-layer
// forward (H_1' = relu(X' W_1'^T + b_1), schedule and arithmetic of launch_tc_forward):
// h_cur holds this step's batch rows (a.hc_row0 ..), x_next the next step's (a.x_row0 ..).
// W is loaded through w_load (row j / a.w_div) and stored through w_store (row j).
cudaError_t launch_tc_update_forward(const CUtensorMap& w_load, const CUtensorMap& w_store,
                                     const CUtensorMap& h_cur, const CUtensorMap& x_next,
                                     const CUtensorMap& dz, const TcFwdArgs& a, cudaStream_t s);
// Mini-batch fetch for the bf16 path: rows (row0 + b) mod N of X -> H_0.
cudaError_t launch_gather_bf16(const __nv_bfloat16* X, int64_t N, int d0, int B, int Bn,
                               int pitch0, int64_t row0, int P, __nv_bfloat16* H0, cudaStream_t s);
// Softmax cross-entropy gradient of the last layer (bf16 operands out), loss, and
// the SGD update of the last bias.
// b_L is read for learner j at row j / src_div of bias_src and written to row j of bias_L.
cudaError_t launch_xent_bf16(const float* Z, const int32_t* y, int64_t N, int64_t row0, int B,
                             int Bn, int C, int pitch_c, float lr, const float* bias_src,
                             int src_div, float* bias_L, int64_t ld, __nv_bfloat16* dZ,
                             float* loss, int P, cudaStream_t s);

bool head_supported(int C, int in, int B, int P);
cudaError_t head_configure();   // raises the dynamic shared-memory limit once
cudaError_t launch_head(const HeadArgs& a, int P, cudaStream_t s);

// ----------------------------------------------------------------- fp32 CUDA-core step
// Buffers: H_l [P][B][d_l] fp32, Z_L [P][B][d_L], dZ_l [P][B][d_l] fp32.
cudaError_t launch_gather_f32(const float* X, int64_t N, int d0, int B, int64_t row0, int P,
                              float* H0, cudaStream_t s);
cudaError_t launch_fwd_f32(const float* H, const float* W, const float* bias, int64_t ld,
                           int in, int out, int B, int relu, float* out_act, int P,
                           cudaStream_t s);
cudaError_t launch_xent_f32(const float* Z, const int32_t* y, int64_t N, int64_t row0, int B,
                            int C, float* dZ, float* loss, int P, cudaStream_t s);
cudaError_t launch_dx_f32(const float* dZ, const float* W, int64_t ld, const float* Hprev,
                          int in, int out, int B, float* dZprev, int P, cudaStream_t s);
cudaError_t launch_dw_update_f32(const float* dZ, const float* H, float* W, float* bias,
                                 int64_t ld, int in, int out, int B, float lr, int P,
                                 cudaStream_t s);

}  // namespace ha
