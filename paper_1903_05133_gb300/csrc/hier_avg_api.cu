// C ABI of the Hier-AVG hot path (declared in include/hier_avg.h): argument
// validation, the parameter and workspace layout, TMA descriptor construction,
// and the order of kernel launches that makes one local step, one local / global
// average and one round of Algorithm 1 (Sec. 3.1).
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <algorithm>
#include <mutex>
#include <string>
#include <vector>

#include <cuda.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "ptx.cuh"

namespace {

using ha::TcBwdArgs;
using ha::TcFwdArgs;

constexpr int64_t kAlign = 1024;
constexpr int64_t kTargetCtas = 152;   // persistent kernels: one CTA per SM of a GB300
constexpr int64_t kPieceChunks = 48;   // chunks per piece of a split tile (forward, backward)
int64_t round_up(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

struct ProfRec {
  int kind;
  cudaEvent_t a, b;
  double bytes, flops;
};

}  // namespace

struct hier_avg {
  // configuration (Sec. 2 notation)
  int P = 0, S = 0, K1 = 0, K2 = 0, B = 0, L = 0, prec = 0;
  float lr = 0.f;
  int G = 0;                                  // local steps per global round (0: K1 * K2)
  std::vector<int> dims;
  // parameter row layout
  int64_t D = 0, ld = 0;
  std::vector<int64_t> woff, boff;
  // workspace layout
  int Bn = 0;
  std::vector<int> pitch;                       // per width index l = 0..L
  std::vector<int64_t> off_H, off_dZ;
  int64_t off_Z = 0, off_loss = 0, off_err = 0, ws_bytes = 0;
  // Cluster means [P / S, ld] of a compact local average inside a round (bf16 path,
  // S > 1): after the step part of the workspace, which is all a single step needs.
  int64_t off_M = 0, ws_step_bytes = 0;
  bool m_ok = false;                          // the bound workspace holds the means
  // The step that closes a local block inside a round (compact averages only) updates
  // W_1 for groups of upd_group learners of a cluster and stores their adjacent-pair
  // tree sum, to the first learner row of each group through tm_gs[l] (1: not used);
  // the later layers' updates do the same (their dX from a backward without update).
  // grp[l]: the last step stored group sums of W_l.
  int upd_group = 1;
  std::vector<CUtensorMap> tm_gs;
  std::vector<char> grp;
  int64_t off_part = 0, off_cnt = 0;          // stream-K partials and tile counters
  int64_t off_dyn = 0;                        // update kernel's work-item counters
  std::vector<int> fwd_ctas, fwd_tiles;       // per layer: stream-K CTAs, output tiles
  std::vector<int> fwd_cq;                    // per layer: cluster split factor (1 = dynamic)
  std::vector<int> fwd_whole, fwd_np;         // per layer (dynamic): whole tiles, tail pieces
  std::vector<int> fwd_pc;                    // per layer (dynamic): chunks per tail piece
  int fwd_group = 1;                          // learners per grouped forward after an average
  std::vector<int> bwd_ctas, bwd_tiles;       // per layer: CTAs, input slices of 128
  std::vector<int> bwd_whole, bwd_np;         // per layer: whole tiles, tail pieces
  bool fused_xent = false;                    // d_L <= 128: CE in the last forward epilogue
  bool w_stream = true;                       // parameters exceed L2: stream W evict-first
  bool head = false;                          // d_L <= 16: fused last-layer kernel
  // binding
  bool bound = false;
  int device = 0;
  float* params = nullptr;
  uint8_t* ws = nullptr;
  const void* X = nullptr;
  const int32_t* y = nullptr;
  int64_t N = 0;
  cudaStream_t stream = nullptr;
  std::vector<CUtensorMap> tm_wf, tm_wb, tm_h, tm_dz;
  std::vector<CUtensorMap> tm_wf_m, tm_wb_m;  // the same weight views of the cluster means
  CUtensorMap tm_x;                           // X [P][N][d_0] as the first layer's batch tile
  int64_t t = 0;
  int64_t cursor = 0;                         // rows each learner has read (next batch: mod N)
  int Bstep = 0;                              // batch size of the following steps (<= B)
  int64_t launches = 0;                       // kernels launched since bind
  // round_host: the rows of each step are copied on a stream of their own, one step
  // ahead of the kernels, which wait on copied[step]
  cudaStream_t copy_stream = nullptr;
  std::vector<cudaEvent_t> copied;
  cudaEvent_t round_start = nullptr;
  // profiling
  unsigned prof = 0;                          // kinds timed: bit (1 << HA_KERNEL_*)
  int prof_every = 1;                         // time every n-th launch of those kinds
  int64_t prof_seen[HA_KERNEL_KINDS] = {};    // launches of each kind since enabled
  std::vector<ProfRec> recs;
  std::vector<cudaEvent_t> pool;
  size_t pool_used = 0;
  std::string err;

  int fail(int code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    err = buf;
    return code;
  }
  int cuda(cudaError_t e, const char* what) {
    if (e == cudaSuccess) return HA_OK;
    return fail(HA_ECUDA, "%s: %s", what, cudaGetErrorString(e));
  }
  template <class T>
  T* wsp(int64_t off) { return reinterpret_cast<T*>(ws + off); }
  int* err_word() { return wsp<int>(off_err); }
  float* means() { return wsp<float>(off_M); }
  // A word next to the error word that no kernel ever writes (stays zero).
  const int* never_set() { return wsp<int>(off_err) + 1; }
  float* loss() { return wsp<float>(off_loss); }

  cudaEvent_t ev() {
    if (pool_used == pool.size()) {
      cudaEvent_t e;
      if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
      pool.push_back(e);
    }
    return pool[pool_used++];
  }
  // Bracket one launch with events when profiling is on.  bytes and flops: the
  // launch's algorithmic memory traffic and arithmetic (multiply-adds count two).
  template <class F>
  int timed(int kind, double bytes, double flops, F&& launch, const char* what) {
    cudaEvent_t a = nullptr, b = nullptr;
    bool on = (prof >> kind) & 1u;
    if (on) on = prof_seen[kind]++ % prof_every == 0;
    ++launches;
    if (on) {
      a = ev();
      b = ev();
      if (a && b) cudaEventRecord(a, stream);
    }
    const cudaError_t e = launch();
    if (e != cudaSuccess) return cuda(e, what);
    if (on && a && b) {
      cudaEventRecord(b, stream);
      recs.push_back({kind, a, b, bytes, flops});
    }
    return HA_OK;
  }
};

namespace {

bool valid_handle(const hier_avg* h) { return h != nullptr; }

int plan_layout(hier_avg* h) {
  const int L = h->L;
  int64_t pos = 0;
  h->woff.assign(L, 0);
  h->boff.assign(L, 0);
  h->D = 0;
  for (int l = 0; l < L; ++l) {
    const int64_t in = h->dims[l], out = h->dims[l + 1];
    h->woff[l] = pos;
    pos = round_up(pos + in * out, 64);
    h->boff[l] = pos;
    pos = round_up(pos + out, 64);
    h->D += in * out + out;
  }
  h->ld = round_up(pos, 64);

  const int64_t P = h->P, B = h->B;
  int64_t off = 0;
  auto take = [&](int64_t bytes) {
    const int64_t o = off;
    off = round_up(off + bytes, kAlign);
    return o;
  };
  h->off_H.assign(L + 1, 0);
  h->off_dZ.assign(L + 1, 0);
  h->pitch.assign(L + 1, 0);
  if (h->prec == HA_PREC_BF16) {
    h->Bn = static_cast<int>(round_up(B, 16));
    for (int l = 0; l <= L; ++l) h->pitch[l] = static_cast<int>(round_up(h->dims[l], 64));
    for (int l = 0; l < L; ++l) h->off_H[l] = take(P * h->Bn * h->pitch[l] * 2);
    for (int l = 1; l <= L; ++l) h->off_dZ[l] = take(P * h->Bn * h->pitch[l] * 2);
    // Stream-K plans of the forward and backward GEMMs: at most one persistent CTA
    // per SM of a GB300 (152).  They depend on the shapes only, so the summation
    // order of split tiles is the same on every GPU.  Forward tile = 128 outputs x
    // 64-input chunks; backward tile = 128 inputs x 64-output chunks.
    h->fwd_group = h->S > 1 ? ha::tc_forward_group_size(h->S, h->Bn) : 1;
    h->fwd_ctas.assign(L, 1);
    h->fwd_tiles.assign(L, 1);
    h->fwd_cq.assign(L, 1);
    h->fwd_whole.assign(L, 0);
    h->fwd_np.assign(L, 1);
    h->fwd_pc.assign(L, static_cast<int>(kPieceChunks));
    h->bwd_ctas.assign(L, 1);
    h->bwd_tiles.assign(L, 1);
    h->bwd_whole.assign(L, 0);
    h->bwd_np.assign(L, 1);
    int64_t part_bytes = 16, max_tiles = 1;
    for (int l = 0; l < L; ++l) {
      const int64_t in = h->dims[l], out = h->dims[l + 1];
      const int64_t ftiles = (out + 127) / 128, btiles = (in + 127) / 128;
      h->fwd_tiles[l] = static_cast<int>(ftiles);
      // Few tiles: a cluster of cq CTAs per tile, reduced through distributed shared
      // memory (the stream-K fix-up through global memory costs a few microseconds of
      // latency at the end, which is a large share of a short layer).
      const int64_t nk = (in + 63) / 64;
      const int64_t cq = std::min<int64_t>(std::min<int64_t>(8, nk), kTargetCtas / (ftiles * P));
      if (cq >= 2) {
        h->fwd_cq[l] = static_cast<int>(cq);
        h->fwd_ctas[l] = static_cast<int>(ftiles * P * cq);
      } else {
        // Dynamic items.  First layer: the last tiles, one per SM, are split into pieces
        // of kPieceChunks chunks, so that the work left when the whole tiles run out is
        // fine grained (the update+forward kernel, which streams W_1 twice as long as a
        // forward, gains most).  The split depends on the shapes only, so the forward
        // and the update+forward sum every H_1 entry the same way.  Later layers keep
        // whole tiles: there a piece's partial round trip costs more than the balance
        // gains (measured).
        // (With groups of G learners forwarded together after a compact average, the
        // tail is rounded down to whole groups, at least one: the grouped kernel splits
        // the same tiles.  Rounding up measured slightly slower.)
        const int64_t gt = h->fwd_group * ftiles;
        const int64_t t_tail =
            l == 0 ? std::min<int64_t>(ftiles * P, std::max<int64_t>(gt, kTargetCtas / gt * gt)) : 0;
        const int64_t pc = h->fwd_pc[l];
        const int64_t np = (nk + pc - 1) / pc;
        h->fwd_whole[l] = static_cast<int>(ftiles * P - t_tail);
        h->fwd_np[l] = static_cast<int>(np);
        const int64_t items = (ftiles * P - t_tail) + t_tail * np;
        h->fwd_ctas[l] = static_cast<int>(std::min<int64_t>(kTargetCtas, items));
        if (np > 1) part_bytes = std::max(part_bytes, t_tail * np * 128 * h->Bn * 4);
      }
      {
        // Backward with dX (every layer but the first; the first runs the update-only
        // kernel): dynamic items, the last tiles (one per SM) split into pieces whose dX
        // partials are added in piece order.  (A tail of whole learners, which would let
        // the learners of a cluster claim the pieces with the same rows of the cluster
        // mean together after an average, balanced every step worse: 3072-2048-2048-10
        // backward 357 -> 361 us per launch.)
        const int64_t nc = (out + 63) / 64;
        const int64_t t_tail = std::min<int64_t>(btiles * P, kTargetCtas);
        const int64_t np = (nc + kPieceChunks - 1) / kPieceChunks;
        h->bwd_whole[l] = static_cast<int>(btiles * P - t_tail);
        h->bwd_np[l] = static_cast<int>(np);
        h->bwd_ctas[l] = static_cast<int>(
            std::min<int64_t>(kTargetCtas, (btiles * P - t_tail) + t_tail * np));
        if (l > 0 && np > 1) part_bytes = std::max(part_bytes, t_tail * np * 128 * h->Bn * 4);
      }
      h->bwd_tiles[l] = static_cast<int>(btiles);
      max_tiles = std::max(max_tiles, std::max(ftiles, btiles) * P);
    }
    h->fused_xent = h->dims[L] <= 128;
    h->head = ha::head_supported(h->dims[L], h->dims[L - 1], static_cast<int>(B), h->P);
    h->off_part = take(part_bytes);
    h->off_cnt = take(max_tiles * 4);
    h->off_dyn = take(16);
  } else {
    for (int l = 0; l <= L; ++l) h->pitch[l] = h->dims[l];
    for (int l = 0; l < L; ++l) h->off_H[l] = take(P * B * h->dims[l] * 4);
    for (int l = 1; l <= L; ++l) h->off_dZ[l] = take(P * B * h->dims[l] * 4);
  }
  h->off_Z = take(P * B * h->dims[L] * 4);
  h->off_loss = take(P * 4);
  h->off_err = take(16);
  h->ws_step_bytes = off;
  if (h->prec == HA_PREC_BF16 && h->S > 1) h->off_M = take((P / h->S) * h->ld * 4);
  h->ws_bytes = off;
  return HA_OK;
}

int make_map(hier_avg* h, CUtensorMap* m, CUtensorMapDataType dt, void* base, uint64_t d0,
             uint64_t d1, uint64_t d2, uint64_t s1_bytes, uint64_t s2_bytes, uint32_t b0,
             uint32_t b1, CUtensorMapSwizzle sw) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return h->fail(HA_ECUDA, "cuTensorMapEncodeTiled is unavailable");
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {s1_bytes, s2_bytes};
  const cuuint32_t box[3] = {b0, b1, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  const CUresult r = enc(m, dt, 3, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                         sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return h->fail(HA_ECUDA, "cuTensorMapEncodeTiled failed (%d) for dims %llu x %llu x %llu",
                   static_cast<int>(r), (unsigned long long)d0, (unsigned long long)d1,
                   (unsigned long long)d2);
  return HA_OK;
}

int build_maps(hier_avg* h) {
  const int L = h->L;
  // When all learners' parameters fit in L2, the backward re-reads what the
  // forward just read and the next step what the backward wrote, so W keeps the
  // normal L2 policy; otherwise it is marked evict-first so that it does not push
  // the small, re-read activation tiles out of L2.
  int l2 = 0;
  if (cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, h->device) != cudaSuccess) l2 = 0;
  h->w_stream = static_cast<double>(h->P) * h->ld * 4 > static_cast<double>(l2);
  h->tm_wf.resize(L);
  h->tm_wb.resize(L);
  h->tm_wf_m.resize(h->m_ok ? L : 0);
  h->tm_gs.resize(L);
  h->tm_wb_m.resize(h->m_ok ? L : 0);
  h->tm_h.resize(L);
  h->tm_dz.resize(L + 1);
  const uint64_t P = h->P, Bn = h->Bn;
  int rc;
  for (int l = 0; l < L; ++l) {
    const uint64_t in = h->dims[l], out = h->dims[l + 1];
    float* W = h->params + h->woff[l];
    if ((rc = make_map(h, &h->tm_wf[l], CU_TENSOR_MAP_DATA_TYPE_FLOAT32, W, in, out, P, in * 4,
                       h->ld * 4, 32, 128, CU_TENSOR_MAP_SWIZZLE_128B)))
      return rc;
    if ((rc = make_map(h, &h->tm_wb[l], CU_TENSOR_MAP_DATA_TYPE_FLOAT32, W, in, out, P, in * 4,
                       h->ld * 4, 128, 64, CU_TENSOR_MAP_SWIZZLE_NONE)))
      return rc;
    if (h->m_ok && h->upd_group > 1) {
      // group sums of W_l: row g*Q of the parameter matrix, g < P / Q
      const uint64_t Q = h->upd_group;
      if ((rc = make_map(h, &h->tm_gs[l], CU_TENSOR_MAP_DATA_TYPE_FLOAT32, W, in, out, P / Q, in * 4,
                         Q * h->ld * 4, 128, 64, CU_TENSOR_MAP_SWIZZLE_NONE)))
        return rc;
    }
    if (h->m_ok) {
      float* Wm = h->means() + h->woff[l];
      const uint64_t G = P / h->S;
      if ((rc = make_map(h, &h->tm_wf_m[l], CU_TENSOR_MAP_DATA_TYPE_FLOAT32, Wm, in, out, G, in * 4,
                         h->ld * 4, 32, 128, CU_TENSOR_MAP_SWIZZLE_128B)))
        return rc;
      if ((rc = make_map(h, &h->tm_wb_m[l], CU_TENSOR_MAP_DATA_TYPE_FLOAT32, Wm, in, out, G, in * 4,
                         h->ld * 4, 128, 64, CU_TENSOR_MAP_SWIZZLE_NONE)))
        return rc;
    }
    const uint64_t pin = h->pitch[l];
    if ((rc = make_map(h, &h->tm_h[l], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, h->ws + h->off_H[l], pin,
                       Bn, P, pin * 2, Bn * pin * 2, 64, static_cast<uint32_t>(Bn),
                       CU_TENSOR_MAP_SWIZZLE_128B)))
      return rc;
  }
  {
    const uint64_t d0 = h->dims[0], N = h->N;
    if ((rc = make_map(h, &h->tm_x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, const_cast<void*>(h->X), d0,
                       N, P, d0 * 2, N * d0 * 2, 64, static_cast<uint32_t>(Bn),
                       CU_TENSOR_MAP_SWIZZLE_128B)))
      return rc;
  }
  for (int l = 1; l <= L; ++l) {
    const uint64_t d = h->dims[l], pd = h->pitch[l];
    if ((rc = make_map(h, &h->tm_dz[l], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, h->ws + h->off_dZ[l], pd,
                       Bn, P, pd * 2, Bn * pd * 2, 64, static_cast<uint32_t>(Bn),
                       CU_TENSOR_MAP_SWIZZLE_128B)))
      return rc;
  }
  return HA_OK;
}

int check_bound(hier_avg* h) {
  if (!h) return HA_EINVAL;
  if (!h->bound) return h->fail(HA_ESTATE, "hier_avg_bind has not been called");
  return HA_OK;
}

// Makes a device current for the lifetime of the object and gives the calling
// thread its previous current device back afterwards, so that no entry point
// changes the caller's device.
class DeviceScope {
 public:
  explicit DeviceScope(int device) {
    if (cudaGetDevice(&prev_) == cudaSuccess && prev_ != device)
      changed_ = cudaSetDevice(device) == cudaSuccess;
  }
  ~DeviceScope() {
    if (changed_) cudaSetDevice(prev_);
  }
  DeviceScope(const DeviceScope&) = delete;
  DeviceScope& operator=(const DeviceScope&) = delete;

 private:
  int prev_ = 0;
  bool changed_ = false;
};

// Algorithmic bytes of the big kernels (fp32 master read + write, activations).
double bytes_forward(const hier_avg* h, int l) {
  const double P = h->P, in = h->dims[l], out = h->dims[l + 1], B = h->Bstep;
  const double act = h->prec == HA_PREC_BF16 ? 2.0 : 4.0;
  return P * (in * out * 4.0 + out * 4.0 + B * in * act + B * out * (l + 1 == h->L ? 4.0 : act));
}
// The first layer's update fused with the next step's first-layer forward: W read and
// written once, this step's and the next step's batch rows, dZ_1 read, b_1 read, H_1' written.
double bytes_update_forward(const hier_avg* h) {
  const double P = h->P, in = h->dims[0], out = h->dims[1], B = h->Bstep;
  return P * (in * out * 8.0 + out * 4.0 + 2.0 * B * in * 2.0 + 2.0 * B * out * 2.0);
}
double bytes_backward(const hier_avg* h, int l) {
  const double P = h->P, in = h->dims[l], out = h->dims[l + 1], B = h->Bstep;
  const double act = h->prec == HA_PREC_BF16 ? 2.0 : 4.0;
  const double dx = l > 0 ? (B * in * act + in * 8.0) : 0.0;
  return P * (in * out * 8.0 + B * in * act + B * out * act + dx);
}

// Right after a compact local average the S learners of a cluster read one row of
// means: the weights of layer l count once per cluster, not once per learner.
double shared_w_bytes(const hier_avg* h, int l, bool means) {
  if (!means) return 0.0;
  return double(h->P) * h->dims[l] * h->dims[l + 1] * 4.0 * (1.0 - 1.0 / h->S);
}

// Algorithmic flops of the learner-step products (2 per multiply-add): one
// [B x in] x [in x out] product per learner for the forward, dW and dX each.
double flops_gemm(const hier_avg* h, int l) {
  return 2.0 * h->P * h->Bstep * double(h->dims[l]) * h->dims[l + 1];
}

// Arguments of the small last layer (input H_{L-1}, or X rows for a one-layer model).
// Where a step reads the parameters from: learner j's own row (div 1), or, in the
// first step after a compact local average, row j / S of the cluster means.
struct ParamSrc {
  const float* base;
  int div;
};
ParamSrc param_src(hier_avg* h, bool means) {
  return means ? ParamSrc{h->means(), h->S} : ParamSrc{h->params, 1};
}

ha::HeadArgs head_args(hier_avg* h, ParamSrc src) {
  const int L = h->L;
  ha::HeadArgs a{};
  a.C = h->dims[L];
  a.in = h->dims[L - 1];
  a.B = h->Bstep;
  a.Bn = h->Bn;
  a.pitch_in = h->pitch[L - 1];
  a.ld = h->ld;
  a.N = h->N;
  a.row0 = h->cursor % h->N;
  a.lr = h->lr;
  a.W = h->params + h->woff[L - 1];
  a.bias = h->params + h->boff[L - 1];
  a.W_src = src.base + h->woff[L - 1];
  a.bias_src = src.base + h->boff[L - 1];
  a.src_div = src.div;
  a.x_rows = L == 1;
  a.H = L == 1 ? static_cast<const __nv_bfloat16*>(h->X) : h->wsp<__nv_bfloat16>(h->off_H[L - 1]);
  a.y = h->y;
  a.has_dx = L > 1;
  if (L > 1) {
    a.bias_prev = h->params + h->boff[L - 2];
    a.bias_prev_src = src.base + h->boff[L - 2];
    a.dz_prev = h->wsp<__nv_bfloat16>(h->off_dZ[L - 1]);
  }
  a.loss = h->loss();
  return a;
}

// One step.  h1_ready: H_1 of this step was written by the previous step's
// update+forward kernel (skip the first layer's forward).  fuse_next: the caller runs
// the next step right after this one with nothing in between, so this step may
// compute the next step's H_1; *fused reports whether it did.  from_means: the caller
// has just taken a compact local average (do_local_means), so every learner's
// parameters are its cluster's mean: every kernel reads them from row j / S of the
// means and writes learner j's own row.  Every weight and bias is updated exactly once
// per step, so after this step every learner row holds its parameters again.
// next_rows (round_host): recorded once the next step's rows are on the device; the
// update+forward kernel, which reads them, waits for it.
// group_out: a local average follows this step (compact, or fused with the global
// average) and reads the round's means; the weight updates of the tensor-core layers may
// then store group sums of W_l (h->upd_group learners each) instead of the learner rows'
// W_l, and h->grp[l] records which did (the average must then read them).
int do_step(hier_avg* h, bool h1_ready = false, bool fuse_next = false, bool* fused = nullptr,
            bool from_means = false, cudaEvent_t next_rows = nullptr, bool group_out = false) {
  const int L = h->L, P = h->P, B = h->Bstep;
  if (fused) *fused = false;
  h->grp.assign(L, 0);
  const int q = group_out && h->m_ok ? h->upd_group : 1;
  cudaStream_t s = h->stream;
  int rc;
  const bool means = from_means && h->m_ok;
  const ParamSrc src = param_src(h, means);
  if (h->prec == HA_PREC_BF16) {
    const int d0 = h->dims[0];
    // The first layer reads its batch tile straight from X unless the batch wraps
    // around the end of the data set; then the rows are gathered first.
    const int64_t r0 = h->cursor % h->N;   // this step's batch: rows r0 .. (mod N)
    const bool x_direct = r0 + B <= h->N;
    if (!x_direct) {
      rc = h->timed(HA_KERNEL_GATHER, double(P) * B * d0 * 2 * 3, 0.0, [&] {
        return ha::launch_gather_bf16(static_cast<const __nv_bfloat16*>(h->X), h->N, d0, B, h->Bn,
                                      h->pitch[0], r0, P, h->wsp<__nv_bfloat16>(h->off_H[0]), s);
      }, "gather");
      if (rc) return rc;
    }
    const int n_fwd = h->head ? L - 1 : L;
    for (int l = h1_ready ? 1 : 0; l < n_fwd; ++l) {
      TcFwdArgs a{};
      a.in = h->dims[l];
      a.out = h->dims[l + 1];
      a.B = B;
      a.Bn = h->Bn;
      a.ld = h->ld;
      a.bias = src.base + h->boff[l];
      a.b_div = src.div;
      a.w_div = src.div;
      a.bias_out = h->params + h->boff[l];
      a.ctas = h->fwd_ctas[l];
      a.cq = h->fwd_cq[l];
      a.o_tiles = h->fwd_tiles[l];
      a.n_tiles = h->fwd_tiles[l] * P;
      a.n_whole = h->fwd_whole[l];
      a.np_tail = h->fwd_np[l];
      a.piece_chunks = h->fwd_pc[l];
      a.part = h->wsp<float>(h->off_part);
      a.counters = h->wsp<int>(h->off_cnt);
      a.dyn = h->wsp<int>(h->off_dyn);
      a.x_direct = (l == 0 && x_direct) ? 1 : 0;
      a.w_stream = h->w_stream ? 1 : 0;
      a.x_row0 = static_cast<int>(r0);
      if (l + 1 < L) {
        a.mode = 0;
        a.h_out = h->wsp<__nv_bfloat16>(h->off_H[l + 1]);
        a.pitch_out = h->pitch[l + 1];
      } else if (h->fused_xent) {
        a.mode = 2;
        a.y = h->y;
        a.N = h->N;
        a.row0 = r0;
        a.lr = h->lr;
        a.pitch_out = h->pitch[L];
        a.dz_out = h->wsp<__nv_bfloat16>(h->off_dZ[L]);
        a.loss = h->loss();
      } else {
        a.mode = 1;
        a.z_out = h->wsp<float>(h->off_Z);
      }
      a.err = h->err_word();
      const CUtensorMap& hin = a.x_direct ? h->tm_x : h->tm_h[l];
      // Right after a compact local average: groups of G learners of a cluster share the
      // cluster mean's weights, forwarded as one product per weight tile.
      const int G = h->fwd_group;
      if (means && G > 1 && a.cq == 1 && a.mode != 2 && a.n_whole % (G * a.o_tiles) == 0) {
        const int gw = a.n_whole / G;
        a.ctas = static_cast<int>(std::min<int64_t>(kTargetCtas, gw + int64_t(a.n_tiles / G - gw) * a.np_tail));
        rc = h->timed(HA_KERNEL_FORWARD, bytes_forward(h, l) - shared_w_bytes(h, l, true),
                      flops_gemm(h, l), [&] {
          return ha::launch_tc_forward_group(h->tm_wf_m[l], hin, a, G, s);
        }, "forward");
      } else {
        rc = h->timed(HA_KERNEL_FORWARD, bytes_forward(h, l) - shared_w_bytes(h, l, means),
                      flops_gemm(h, l), [&] {
          return ha::launch_tc_forward(means ? h->tm_wf_m[l] : h->tm_wf[l], hin, a, P, s);
        }, "forward");
      }
      if (rc) return rc;
    }
    const int C = h->dims[L];
    if (h->head) {
      const ha::HeadArgs a = head_args(h, src);
      const double hb = double(P) * (8.0 * C * a.in + 2.0 * B * a.in * 2 + (L > 1 ? 4.0 * B * a.in : 0)) -
                        shared_w_bytes(h, L - 1, means);
      const double hf = flops_gemm(h, L - 1) * (L > 1 ? 3 : 2);   // forward, dW (, dX)
      rc = h->timed(HA_KERNEL_HEAD, hb, hf, [&] { return ha::launch_head(a, P, s); }, "head");
      if (rc) return rc;
    } else if (!h->fused_xent) {
      rc = h->timed(HA_KERNEL_XENT, double(P) * B * C * 4 * 3, 0.0, [&] {
        return ha::launch_xent_bf16(h->wsp<float>(h->off_Z), h->y, h->N, r0, B, h->Bn, C,
                                    h->pitch[L], h->lr, src.base + h->boff[L - 1], src.div,
                                    h->params + h->boff[L - 1], h->ld,
                                    h->wsp<__nv_bfloat16>(h->off_dZ[L]), h->loss(), P, s);
      }, "xent");
      if (rc) return rc;
    }
    for (int l = h->head ? L - 2 : L - 1; l >= 0; --l) {
      TcBwdArgs a{};
      a.in = h->dims[l];
      a.out = h->dims[l + 1];
      a.B = B;
      a.Bn = h->Bn;
      a.ld = h->ld;
      a.lr = h->lr;
      a.has_dx = l > 0;
      a.src_div = src.div;
      if (a.has_dx) {
        a.bias_prev = h->params + h->boff[l - 1];
        a.bias_prev_src = src.base + h->boff[l - 1];
        a.dz_prev = h->wsp<__nv_bfloat16>(h->off_dZ[l]);
        a.pitch_in = h->pitch[l];
      }
      const CUtensorMap& wl = means ? h->tm_wb_m[l] : h->tm_wb[l];   // W read ...
      const CUtensorMap& ws = h->tm_wb[l];                           // ... and written
      // H_{l-1}: the layer's input rows, straight from X for the first layer when
      // the forward read them there too.
      const bool from_x = l == 0 && x_direct;
      a.h_row0 = from_x ? static_cast<int>(r0) : 0;
      a.w_stream = h->w_stream ? 1 : 0;
      a.ctas = h->bwd_ctas[l];
      a.s_tiles = h->bwd_tiles[l];
      a.n_tiles = h->bwd_tiles[l] * P;
      a.n_whole = h->bwd_whole[l];
      a.np_tail = h->bwd_np[l];
      a.piece_chunks = static_cast<int>(kPieceChunks);
      a.dyn = h->wsp<int>(h->off_dyn);
      a.part = h->wsp<float>(h->off_part);
      a.counters = h->wsp<int>(h->off_cnt);
      a.err = h->err_word();
      const CUtensorMap& hin = from_x ? h->tm_x : h->tm_h[l];
      // The next step's batch, if contiguous in X, lets the first layer's update also
      // produce the next step's H_1 (the layer must be hidden, i.e. L >= 2).
      const int64_t r1 = (h->cursor + B) % h->N;
      if (l == 0 && fuse_next && L >= 2 && r1 + B <= h->N) {
        TcFwdArgs f{};
        f.in = h->dims[0];
        f.out = h->dims[1];
        f.B = B;
        f.Bn = h->Bn;
        f.ld = h->ld;
        f.bias = h->params + h->boff[0];   // b_1 after this step's update (row j)
        f.b_div = 1;
        f.w_div = src.div;                 // W_1 before it (from the means after an average)
        f.mode = 0;
        f.h_out = h->wsp<__nv_bfloat16>(h->off_H[1]);
        f.pitch_out = h->pitch[1];
        f.ctas = h->fwd_ctas[0];
        f.cq = h->fwd_cq[0];
        f.o_tiles = h->fwd_tiles[0];
        f.n_tiles = h->fwd_tiles[0] * P;
        f.n_whole = h->fwd_whole[0];
        f.np_tail = h->fwd_np[0];
        f.piece_chunks = h->fwd_pc[0];
        f.part = h->wsp<float>(h->off_part);
        f.counters = h->wsp<int>(h->off_cnt);
        f.dyn = h->wsp<int>(h->off_dyn);
        f.x_direct = 1;
        f.x_row0 = static_cast<int>(r1);
        f.hc_row0 = a.h_row0;
        f.w_stream = a.w_stream;
        f.lr = h->lr;
        f.err = h->err_word();
        if (next_rows && (rc = h->cuda(cudaStreamWaitEvent(s, next_rows, 0), "round_host: wait for the rows")))
          return rc;
        rc = h->timed(HA_KERNEL_UPDATE_FORWARD, bytes_update_forward(h) - shared_w_bytes(h, 0, means),
                      2 * flops_gemm(h, 0), [&] {
          return ha::launch_tc_update_forward(means ? h->tm_wf_m[0] : h->tm_wf[0], h->tm_wf[0], hin,
                                              h->tm_x, h->tm_dz[1], f, s);
        }, "update+forward");
        if (rc) return rc;
        if (fused) *fused = true;
        continue;
      }
      // The first layer's backward (no dX) runs the update-only kernel: independent
      // runs of 8 chunks, claimed dynamically (measured faster than the backward
      // kernel's items for short layers too: 3072-512-10 round 0.859 -> 0.850 ms).
      // Grouped (q > 1): W_l read per learner, its group sums written to row g*q of the
      // W_l region, g < P / q.  A layer with dX first runs the backward without update
      // (dZ_{l-1}, b_{l-1}), which reads W_l once more: worth it for quads only (per
      // weight and learner 4 more bytes read, 2 * (4 - 4 / q) fewer moved by the update
      // and the average; pairs measured slower, 3072-2048-2048-10 36.02 -> 36.21 ms).
      const double wbytes = double(P) * h->dims[l] * h->dims[l + 1] * 4.0;
      const int ql = a.has_dx && q < 4 ? 1 : q;
      const double gb = ql > 1 ? wbytes * (1.0 - 1.0 / ql) : 0.0;
      if (a.has_dx && ql > 1) {
        a.no_update = 1;
        rc = h->timed(HA_KERNEL_BACKWARD, bytes_backward(h, l) - wbytes - shared_w_bytes(h, l, means),
                      flops_gemm(h, l), [&] {
          return ha::launch_tc_backward(wl, ws, hin, h->tm_dz[l + 1], a, P, s);
        }, "backward");
        if (rc) return rc;
        a.no_update = 0;
        a.has_dx = 0;
      }
      if (a.has_dx) {
        rc = h->timed(HA_KERNEL_BACKWARD, bytes_backward(h, l) - shared_w_bytes(h, l, means),
                      flops_gemm(h, l) * 2, [&] {
          return ha::launch_tc_backward(wl, ws, hin, h->tm_dz[l + 1], a, P, s);
        }, "backward");
      } else {
        a.ctas = kTargetCtas;
        const double ub = double(P) * (h->dims[l] * h->dims[l + 1] * 8.0 + double(B) * h->dims[l] * 2 +
                                       double(B) * h->dims[l + 1] * 2);
        rc = h->timed(HA_KERNEL_BACKWARD, ub - gb - shared_w_bytes(h, l, means), flops_gemm(h, l), [&] {
          return ha::launch_tc_update(wl, ql > 1 ? h->tm_gs[l] : ws, hin, h->tm_dz[l + 1], a, ql, s);
        }, "backward");
        h->grp[l] = ql > 1;
      }
      if (rc) return rc;
    }
  } else {
    const int d0 = h->dims[0];
    rc = h->timed(HA_KERNEL_GATHER, double(P) * B * d0 * 4 * 2, 0.0, [&] {
      return ha::launch_gather_f32(static_cast<const float*>(h->X), h->N, d0, B, h->cursor % h->N, P,
                                   h->wsp<float>(h->off_H[0]), s);
    }, "gather");
    if (rc) return rc;
    for (int l = 0; l < L; ++l) {
      const bool last = l + 1 == L;
      float* outp = last ? h->wsp<float>(h->off_Z) : h->wsp<float>(h->off_H[l + 1]);
      rc = h->timed(HA_KERNEL_FORWARD, bytes_forward(h, l), flops_gemm(h, l), [&] {
        return ha::launch_fwd_f32(h->wsp<float>(h->off_H[l]), h->params + h->woff[l],
                                  h->params + h->boff[l], h->ld, h->dims[l], h->dims[l + 1], B,
                                  last ? 0 : 1, outp, P, s);
      }, "forward");
      if (rc) return rc;
    }
    rc = h->timed(HA_KERNEL_XENT, double(P) * B * h->dims[L] * 4 * 2, 0.0, [&] {
      return ha::launch_xent_f32(h->wsp<float>(h->off_Z), h->y, h->N, h->cursor % h->N, B, h->dims[L],
                                 h->wsp<float>(h->off_dZ[L]), h->loss(), P, s);
    }, "xent");
    if (rc) return rc;
    for (int l = L - 1; l >= 0; --l) {
      rc = h->timed(HA_KERNEL_BACKWARD, bytes_backward(h, l), flops_gemm(h, l) * (l > 0 ? 2 : 1), [&] {
        cudaError_t e = cudaSuccess;
        if (l > 0) ++h->launches;   // dX is its own launch
        if (l > 0)
          e = ha::launch_dx_f32(h->wsp<float>(h->off_dZ[l + 1]), h->params + h->woff[l], h->ld,
                                h->wsp<float>(h->off_H[l]), h->dims[l], h->dims[l + 1], B,
                                h->wsp<float>(h->off_dZ[l]), P, s);
        if (e != cudaSuccess) return e;
        return ha::launch_dw_update_f32(h->wsp<float>(h->off_dZ[l + 1]), h->wsp<float>(h->off_H[l]),
                                        h->params + h->woff[l], h->params + h->boff[l], h->ld,
                                        h->dims[l], h->dims[l + 1], B, h->lr, P, s);
      }, "backward");
      if (rc) return rc;
    }
  }
  ++h->t;
  h->cursor += B;
  return HA_OK;
}

int do_local(hier_avg* h) {
  return h->timed(HA_KERNEL_LOCAL_AVG, 8.0 * h->P * h->ld, double(h->P) * h->ld, [&] {
    return ha::launch_group_mean(h->params, h->P, h->S, h->ld, h->ld, h->stream);
  }, "local average");
}

// The local average inside a round, written compactly: each cluster's mean once, to
// row g of the means [P / S, ld], instead of to its S learner rows.  The next step
// reads every learner's parameters from there (do_step's from_means) and writes the
// learner rows, so the values every kernel sees are those of the full write-back.
// Algorithmic bytes: P rows read, P / S rows written.
int do_local_means(hier_avg* h) {
  return h->timed(HA_KERNEL_LOCAL_AVG, 4.0 * h->P * h->ld + 4.0 * (h->P / h->S) * h->ld,
                  double(h->P) * h->ld, [&] {
    return ha::launch_group_mean_to(h->params, h->P, h->S, h->ld, h->ld, h->means(), h->stream);
  }, "local average");
}

// The parameter row in column ranges for an average after a grouped step: the W_l
// regions whose group sums the step stored (h->grp[l]) and the ranges between them
// (biases, padding, the other layers' weights), read from the learner rows.
struct AvgRange {
  int64_t c0, c1;
  bool grouped;
};
std::vector<AvgRange> avg_ranges(const hier_avg* h) {
  std::vector<AvgRange> r;
  int64_t c = 0;
  for (int l = 0; l < h->L; ++l) {
    if (!h->grp[l]) continue;
    const int64_t w0 = h->woff[l], w1 = w0 + static_cast<int64_t>(h->dims[l]) * h->dims[l + 1];
    if (w0 > c) r.push_back({c, w0, false});
    r.push_back({w0, w1, true});
    c = w1;
  }
  if (c < h->ld) r.push_back({c, h->ld, false});
  return r;
}

// The compact local average after a grouped step: each grouped W_l from its group sums
// (rows g*Q, g < P / Q, which hold the first log2(Q) levels of every cluster's
// adjacent-pair tree), the rest of the row from the learner rows.  The tree over a
// cluster's S / Q group sums has the same levels above them as the tree over its S
// rows (Q divides S, so every group is a complete, aligned sub-tree), so the means
// are the bits of do_local_means.
int do_local_means_grouped(hier_avg* h) {
  const int64_t P = h->P, S = h->S, Q = h->upd_group, ld = h->ld;
  const std::vector<AvgRange> rs = avg_ranges(h);
  double bytes = 4.0 * (P / S) * ld;
  for (const AvgRange& r : rs) bytes += 4.0 * (r.grouped ? P / Q : P) * (r.c1 - r.c0);
  return h->timed(HA_KERNEL_LOCAL_AVG, bytes, double(P) * ld, [&] {
    h->launches += static_cast<int64_t>(rs.size()) - 1;   // one launch per range
    for (const AvgRange& r : rs) {
      const cudaError_t e =
          r.grouped ? ha::launch_group_sum_mean_to(h->params + r.c0, P / Q, S / Q, r.c1 - r.c0, Q * ld,
                                                   static_cast<float>(S), h->means() + r.c0, ld, h->stream)
                    : ha::launch_group_mean_to(h->params + r.c0, P, S, r.c1 - r.c0, ld,
                                               h->means() + r.c0, h->stream);
      if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
  }, "local average");
}

int do_local_global(hier_avg* h) {
  return h->timed(HA_KERNEL_GLOBAL_AVG, 8.0 * h->P * h->ld, double(h->P) * h->ld, [&] {
    return ha::launch_local_global_mean(h->params, h->P, h->S, h->ld, h->ld, h->stream);
  }, "local+global average");
}

// The fused last local average and global average after a grouped step: grouped W_l
// from their group sums, the rest of the row from the learner rows; every row receives
// the global mean (the bits of do_local_global, as in do_local_means_grouped).
int do_local_global_grouped(hier_avg* h) {
  const int64_t P = h->P, S = h->S, Q = h->upd_group, ld = h->ld;
  const std::vector<AvgRange> rs = avg_ranges(h);
  double bytes = 4.0 * P * ld;
  for (const AvgRange& r : rs) bytes += 4.0 * (r.grouped ? P / Q : P) * (r.c1 - r.c0);
  return h->timed(HA_KERNEL_GLOBAL_AVG, bytes, double(P) * ld, [&] {
    h->launches += static_cast<int64_t>(rs.size()) - 1;   // one launch per range
    for (const AvgRange& r : rs) {
      const cudaError_t e =
          r.grouped ? ha::launch_local_global_from_groups(h->params + r.c0, Q * ld, Q, h->params + r.c0, P,
                                                          S, r.c1 - r.c0, ld, h->stream)
                    : ha::launch_local_global_mean(h->params + r.c0, P, S, r.c1 - r.c0, ld, h->stream);
      if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
  }, "local+global average");
}

int do_global(hier_avg* h) {
  return h->timed(HA_KERNEL_GLOBAL_AVG, 8.0 * h->P * h->ld, double(h->P) * h->ld, [&] {
    return ha::launch_group_mean(h->params, h->P, h->P, h->ld, h->ld, h->stream);
  }, "global average");
}

int round_steps(const hier_avg* h) { return h->G > 0 ? h->G : h->K1 * h->K2; }

// Rows [r0, r0 + n) of every learner's X from host memory.  Spans of at least
// kRowCopySplit bytes per learner go as one contiguous copy per learner when a learner's
// parameter row holds at least kRowCopyMinLd values, so that the P calls (~2.5 us of
// host time each on a fast host) hide behind the kernels of a step; otherwise the span
// goes as one pitched copy for all learners, one call.  (Pitched copies of
// [32][0.75-12.6 MB] spans ran at 190-209 GB/s in one process and at 18 GB/s later in the
// same process, after a few rounds, while per-learner copies of the same spans kept
// 168-184 GB/s.  At 3072-512-10 a step takes ~50 us, and the host's calls are what
// limits its round.)
constexpr int64_t kRowCopySplit = int64_t(512) << 10;
constexpr int64_t kRowCopyMinLd = int64_t(4) << 20;

int copy_rows(hier_avg* h, const void* X_host, int64_t r0, int64_t n, cudaStream_t cs) {
  const int64_t es = h->prec == HA_PREC_BF16 ? 2 : 4;
  const int64_t rowb = static_cast<int64_t>(h->dims[0]) * es;
  uint8_t* X = static_cast<uint8_t*>(const_cast<void*>(h->X));
  const uint8_t* Xh = static_cast<const uint8_t*>(X_host);
  if (n * rowb < kRowCopySplit || h->ld < kRowCopyMinLd)
    return h->cuda(cudaMemcpy2DAsync(X + r0 * rowb, h->N * rowb, Xh + r0 * rowb, h->N * rowb, n * rowb,
                                     h->P, cudaMemcpyHostToDevice, cs), "round_host: X copy");
  for (int j = 0; j < h->P; ++j) {
    const int64_t off = (static_cast<int64_t>(j) * h->N + r0) * rowb;
    if (int rc = h->cuda(cudaMemcpyAsync(X + off, Xh + off, n * rowb, cudaMemcpyHostToDevice, cs),
                         "round_host: X copy"))
      return rc;
  }
  return HA_OK;
}

// Every learner's labels, y_host [P, N] whole, in one contiguous copy (P * N * 4 bytes:
// 0.5 MB for 32 learners of 4096 samples), ahead of the round's rows of X.
int copy_labels(hier_avg* h, const int32_t* y_host, cudaStream_t cs) {
  return h->cuda(cudaMemcpyAsync(const_cast<int32_t*>(h->y), y_host,
                                 static_cast<size_t>(h->P) * h->N * 4, cudaMemcpyHostToDevice, cs),
                 "round_host: y copy");
}

// round_host's row feed: the rows of the round's steps are copied from host memory on
// the library's copy stream in chunks of steps that double in length (step 0, step 1,
// steps 2-3, 4-7, ...).  ensure(k) issues the chunks up to the one holding step k and
// one more, so the copies stay a chunk ahead of the kernels while the host issues only
// 2 P copies per chunk (O(P log G) per round) between kernel launches; event(k) is
// recorded once step k's rows are on the device.
struct RowFeed {
  hier_avg* h;
  const void* X_host;
  int G;
  int issued_to = 0;            // steps [0, issued_to) have their copies issued
  int chunks = 0;
  std::vector<cudaEvent_t> ev;  // ev[k]: event of step k's chunk
  int issue_next() {
    const int k0 = issued_to;
    if (k0 >= G) return HA_OK;
    const int k1 = std::min(G, k0 <= 1 ? k0 + 1 : 2 * k0);
    int64_t r0 = (h->cursor + static_cast<int64_t>(k0) * h->Bstep) % h->N;
    const int64_t rows = static_cast<int64_t>(k1 - k0) * h->Bstep;
    int64_t left = rows < h->N ? rows : h->N;
    if (rows >= h->N) r0 = 0;
    while (left > 0) {
      const int64_t n = (r0 + left <= h->N) ? left : h->N - r0;
      if (int rc = copy_rows(h, X_host, r0, n, h->copy_stream)) return rc;
      left -= n;
      r0 = 0;
    }
    cudaEvent_t e = h->copied[chunks++];
    if (int rc = h->cuda(cudaEventRecord(e, h->copy_stream), "round_host: record")) return rc;
    for (int k = k0; k < k1; ++k) ev[k] = e;
    issued_to = k1;
    return HA_OK;
  }
  int ensure(int k) {
    while (issued_to <= k)
      if (int rc = issue_next()) return rc;
    return issue_next();   // one chunk ahead
  }
};

// One global round (Algorithm 1, Sec. 3.1): G local steps, a local average after every
// K1-th, the global average after the G-th (fused with the local average that closes
// the round when K1 divides G).  G = K1 * K2 unless set: Sec. 3.1 leaves beta = G / K1
// free in practice.  The local averages inside the round are compact (do_local_means)
// when the workspace holds the means; the global average writes every learner row, so
// the round ends with all P rows in place.
// feed (round_host): step k reads the rows of step k and, in an update+forward kernel,
// step k + 1's.  The handle's stream waits for step 0's and step 1's rows before step 0
// (the latter just before step 0's update+forward), then at steps k = 1, 3, 7, ... (k + 1
// a power of two) for the rows up to step 2k + 1, which cover every step until the next
// wait: few waits, since each one ends the overlap of consecutive launches.
int do_round(hier_avg* h, RowFeed* feed = nullptr) {
  int rc;
  const int G = round_steps(h);
  const bool compact = h->m_ok;
  bool h1_ready = false;
  for (int r = 1; r <= G; ++r) {
    const int k = r - 1;
    if (feed && (k == 0 || (k & (k + 1)) == 0)) {
      const int need = k == 0 ? 0 : std::min(2 * k + 1, G - 1);
      if ((rc = feed->ensure(std::max(need, std::min(1, G - 1))))) return rc;
      if ((rc = h->cuda(cudaStreamWaitEvent(h->stream, feed->ev[need], 0), "round_host: wait for the rows")))
        return rc;
    }
    const bool block_end = r % h->K1 == 0;              // a local average follows step r
    const bool after_local = r > 1 && (r - 1) % h->K1 == 0;
    if ((rc = do_step(h, h1_ready, !block_end && r < G, &h1_ready, after_local && compact,
                      feed && r == 1 && G > 1 ? feed->ev[1] : nullptr, compact && block_end)))
      return rc;
    bool grouped = false;
    for (char g : h->grp) grouped = grouped || g;
    if (r < G && block_end &&
        (rc = grouped ? do_local_means_grouped(h) : compact ? do_local_means(h) : do_local(h)))
      return rc;
    if (r == G && block_end) return grouped ? do_local_global_grouped(h) : do_local_global(h);
  }
  return do_global(h);
}

// Failure-detection self-test: the library's two kinds of bounded device wait, each
// on a condition that nothing will ever satisfy.  Thread 0 waits with acquire order
// for a global word to become 1 (it stays 0), then for the first phase of an mbarrier
// that no thread arrives on.  Each wait gives up after `limit` cycles of SM clock and
// records HA_DEVERR_TIMEOUT in the error word; the kernel then returns.  Nothing is in
// flight when it exits (no copy, no MMA), so the context stays usable.
__global__ void k_wait_selftest(const int* never_set, int* err, long long limit) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    ha::mbar_init(&bar, 1);
    ha::fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    ha::spin_acquire_eq(never_set, 1, err, limit);
    ha::mbar_wait(&bar, 0, err, limit);
  }
}

}  // namespace

extern "C" {

const char* hier_avg_strerror(int status) {
  switch (status) {
    case HA_OK: return "ok";
    case HA_EINVAL: return "invalid argument";
    case HA_ENOMEM: return "buffer too small";
    case HA_ECUDA: return "CUDA error";
    case HA_ESTATE: return "call out of order";
    case HA_ETIMEOUT: return "device-side wait timed out";
    case HA_EUNSUPPORTED: return "unsupported configuration";
    default: return "unknown status";
  }
}

const char* hier_avg_last_error(const hier_avg* h) { return h ? h->err.c_str() : "null handle"; }

// groups: how many independent means one launch takes (one per grid row).
static int check_avg_args(const float* w, int64_t P, int64_t S, int64_t D, int64_t ld,
                          int64_t groups) {
  if (P < 1 || S < 1 || P % S != 0 || D < 0 || ld < D) return HA_EINVAL;
  if (D > 0 && !w) return HA_EINVAL;
  if (P > (int64_t(1) << 30) || D > (int64_t(1) << 40)) return HA_EINVAL;
  if (groups > 65535) return HA_EUNSUPPORTED;   // the group index is a grid dimension
  return HA_OK;
}

int hier_avg_local_average_buffer(float* w_dev, int64_t P, int64_t S, int64_t D, int64_t ld,
                                  void* stream) {
  if (int rc = check_avg_args(w_dev, P, S, D, ld, S > 0 ? P / S : 0)) return rc;
  return ha::launch_group_mean(w_dev, P, S, D, ld, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? HA_OK
             : HA_ECUDA;
}

int hier_avg_global_average_buffer(float* w_dev, int64_t P, int64_t D, int64_t ld, void* stream) {
  if (int rc = check_avg_args(w_dev, P, 1, D, ld, 1)) return rc;
  return ha::launch_group_mean(w_dev, P, P, D, ld, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? HA_OK
             : HA_ECUDA;
}

int hier_avg_local_global_average_buffer(float* w_dev, int64_t P, int64_t S, int64_t D,
                                         int64_t ld, void* stream) {
  if (int rc = check_avg_args(w_dev, P, S, D, ld, 1)) return rc;
  return ha::launch_local_global_mean(w_dev, P, S, D, ld, static_cast<cudaStream_t>(stream)) ==
                 cudaSuccess
             ? HA_OK
             : HA_ECUDA;
}

int hier_avg_create(int P, int S, int K1, int K2, float lr, int B, const int* dims, int n_dims,
                    int precision, hier_avg** out) {
  if (!out) return HA_EINVAL;
  *out = nullptr;
  if (P < 1 || S < 1 || K1 < 1 || K2 < 1 || B < 1 || P % S != 0) return HA_EINVAL;
  if (!std::isfinite(lr) || !dims || n_dims < 2 || n_dims > 64) return HA_EINVAL;
  if (precision != HA_PREC_FP32 && precision != HA_PREC_BF16) return HA_EINVAL;
  for (int l = 0; l < n_dims; ++l)
    if (dims[l] < 1 || dims[l] > (1 << 20)) return HA_EINVAL;
  if (P > 65535) return HA_EUNSUPPORTED;   // learner index is a grid dimension
  if (precision == HA_PREC_BF16) {
    if (B > 64) return HA_EUNSUPPORTED;
    for (int l = 0; l + 1 < n_dims; ++l)
      if (dims[l] % 8 != 0) return HA_EUNSUPPORTED;
  }
  hier_avg* h = new (std::nothrow) hier_avg();
  if (!h) return HA_ENOMEM;
  h->P = P;
  h->S = S;
  h->K1 = K1;
  h->K2 = K2;
  h->B = B;
  h->Bstep = B;
  h->lr = lr;
  h->prec = precision;
  h->dims.assign(dims, dims + n_dims);
  h->L = n_dims - 1;
  plan_layout(h);
  *out = h;
  return HA_OK;
}

void hier_avg_destroy(hier_avg* h) {
  if (!h) return;
  for (cudaEvent_t e : h->pool) cudaEventDestroy(e);
  for (cudaEvent_t e : h->copied) cudaEventDestroy(e);
  if (h->round_start) cudaEventDestroy(h->round_start);
  if (h->copy_stream) cudaStreamDestroy(h->copy_stream);
  delete h;
}

int hier_avg_param_layout(const hier_avg* h, int64_t* D, int64_t* ld, int64_t* offsets) {
  if (!valid_handle(h)) return HA_EINVAL;
  if (D) *D = h->D;
  if (ld) *ld = h->ld;
  if (offsets)
    for (int l = 0; l < h->L; ++l) {
      offsets[2 * l] = h->woff[l];
      offsets[2 * l + 1] = h->boff[l];
    }
  return HA_OK;
}

int hier_avg_workspace_bytes(const hier_avg* h, int64_t* bytes) {
  if (!valid_handle(h) || !bytes) return HA_EINVAL;
  *bytes = h->ws_bytes;
  return HA_OK;
}

int hier_avg_bind(hier_avg* h, float* params_dev, void* workspace_dev, int64_t workspace_bytes,
                  const void* X_dev, const int32_t* y_dev, int64_t N, void* stream) {
  if (!h) return HA_EINVAL;
  h->bound = false;
  if (!params_dev || !workspace_dev || !X_dev || !y_dev || N < 1)
    return h->fail(HA_EINVAL, "bind: NULL buffer or N < 1");
  if (reinterpret_cast<uintptr_t>(params_dev) % 256 || reinterpret_cast<uintptr_t>(workspace_dev) % 256)
    return h->fail(HA_EINVAL, "bind: params and workspace must be 256-byte aligned");
  if (h->prec == HA_PREC_BF16 && reinterpret_cast<uintptr_t>(X_dev) % 16)
    return h->fail(HA_EINVAL, "bind: X must be 16-byte aligned");
  if (workspace_bytes < h->ws_bytes)
    return h->fail(HA_ENOMEM, "bind: workspace needs %lld bytes, got %lld",
                   (long long)h->ws_bytes, (long long)workspace_bytes);
  cudaPointerAttributes attr;
  if (cudaPointerGetAttributes(&attr, params_dev) != cudaSuccess || attr.type != cudaMemoryTypeDevice)
    return h->fail(HA_EINVAL, "bind: params is not device memory");
  h->device = attr.device;
  DeviceScope scope(h->device);
  h->params = params_dev;
  h->ws = static_cast<uint8_t*>(workspace_dev);
  h->X = X_dev;
  h->y = y_dev;
  h->N = N;
  h->stream = static_cast<cudaStream_t>(stream);
  h->t = 0;
  h->cursor = 0;
  h->m_ok = h->off_M > 0;
  h->upd_group = 1;
  if (h->m_ok && h->S % 2 == 0 && !(h->head && h->L == 1))
    h->upd_group = h->S % 4 == 0 && ha::tc_update_max_group(h->Bn) >= 4 ? 4 : 2;
  int rc;
  if ((rc = h->cuda(cudaMemsetAsync(h->ws, 0, h->ws_step_bytes, h->stream), "bind: memset"))) return rc;
  if (h->prec == HA_PREC_BF16) {
    if ((rc = h->cuda(ha::tc_configure(), "bind: kernel attributes"))) return rc;
    if ((rc = h->cuda(ha::head_configure(), "bind: kernel attributes"))) return rc;
    if ((rc = build_maps(h))) return rc;
  }
  h->bound = true;
  return HA_OK;
}

int hier_avg_step(hier_avg* h) {
  if (int rc = check_bound(h)) return rc;
  DeviceScope scope(h->device);
  return do_step(h);
}

int hier_avg_local_average(hier_avg* h) {
  if (int rc = check_bound(h)) return rc;
  DeviceScope scope(h->device);
  return do_local(h);
}

int hier_avg_global_average(hier_avg* h) {
  if (int rc = check_bound(h)) return rc;
  DeviceScope scope(h->device);
  return do_global(h);
}

int hier_avg_round(hier_avg* h) {
  if (int rc = check_bound(h)) return rc;
  DeviceScope scope(h->device);
  return do_round(h);
}

int hier_avg_round_host(hier_avg* h, const void* X_host, const int32_t* y_host, float* loss_host) {
  if (int rc = check_bound(h)) return rc;
  DeviceScope scope(h->device);
  if (!X_host || !y_host || !loss_host) return h->fail(HA_EINVAL, "round_host: NULL host buffer");
  const int G = round_steps(h);
  if (!h->copy_stream &&
      h->cuda(cudaStreamCreateWithFlags(&h->copy_stream, cudaStreamNonBlocking), "round_host: stream"))
    return HA_ECUDA;
  if (!h->round_start &&
      h->cuda(cudaEventCreateWithFlags(&h->round_start, cudaEventDisableTiming), "round_host: event"))
    return HA_ECUDA;
  while (static_cast<int>(h->copied.size()) < G) {
    cudaEvent_t e;
    if (int rc = h->cuda(cudaEventCreateWithFlags(&e, cudaEventDisableTiming), "round_host: event")) return rc;
    h->copied.push_back(e);
  }
  int rc;
  if (h->prec != HA_PREC_BF16) {
    // fp32 path: the round's rows (at most two contiguous ranges per learner, at the
    // wrap-around) copied ahead of the round
    const int64_t rows = static_cast<int64_t>(h->Bstep) * G;
    int64_t r0 = h->cursor % h->N, left = rows < h->N ? rows : h->N;
    if (rows >= h->N) r0 = 0;
    if ((rc = copy_labels(h, y_host, h->stream))) return rc;
    while (left > 0) {
      const int64_t n = (r0 + left <= h->N) ? left : h->N - r0;
      if ((rc = copy_rows(h, X_host, r0, n, h->stream))) return rc;
      left -= n;
      r0 = 0;
    }
    if ((rc = do_round(h))) return rc;
  } else {
    // The rows are copied beside the kernels, chunk by chunk (RowFeed).  (Copies of
    // every step issued ahead of the round, 2 P per step, kept the host busy for
    // milliseconds before the first kernel launch: 3072-2048-2048-10 end to end 1.25x
    // the device-resident round.)  The copies start once the work already queued on the
    // handle's stream is done.
    if ((rc = h->cuda(cudaEventRecord(h->round_start, h->stream), "round_host: record")) ||
        (rc = h->cuda(cudaStreamWaitEvent(h->copy_stream, h->round_start, 0), "round_host: wait")) ||
        (rc = copy_labels(h, y_host, h->copy_stream)))
      return rc;
    RowFeed feed{h, X_host, G};
    feed.ev.assign(G, nullptr);
    if ((rc = do_round(h, &feed))) return rc;
  }
  if ((rc = h->cuda(cudaMemcpyAsync(loss_host, h->loss(), h->P * 4, cudaMemcpyDeviceToHost, h->stream),
                    "round_host: loss copy")))
    return rc;
  return hier_avg_check(h);
}

int hier_avg_set_global_steps(hier_avg* h, int steps) {
  if (!h || steps < 0) return HA_EINVAL;
  h->G = steps;
  return HA_OK;
}

int hier_avg_set_batch(hier_avg* h, int B) {
  if (!h || B < 1 || B > h->B) return HA_EINVAL;
  if (B < h->Bstep && h->bound && h->prec == HA_PREC_BF16) {
    // The bf16 path keeps Bn-row gradient tiles; rows from B on must add nothing to dW.
    DeviceScope scope(h->device);
    for (int l = 1; l <= h->L; ++l)
      if (int rc = h->cuda(cudaMemsetAsync(h->ws + h->off_dZ[l], 0,
                                           static_cast<size_t>(h->P) * h->Bn * h->pitch[l] * 2,
                                           h->stream), "set_batch: clear dZ"))
        return rc;
  }
  h->Bstep = B;
  return HA_OK;
}

int hier_avg_set_lr(hier_avg* h, float lr) {
  if (!h || !std::isfinite(lr)) return HA_EINVAL;
  h->lr = lr;
  return HA_OK;
}

int hier_avg_get_step(const hier_avg* h, int64_t* t) {
  if (!h || !t) return HA_EINVAL;
  *t = h->t;
  return HA_OK;
}

int hier_avg_set_step(hier_avg* h, int64_t t) {
  if (!h || t < 0) return HA_EINVAL;
  h->t = t;
  h->cursor = t * h->Bstep;
  return HA_OK;
}

int hier_avg_losses(hier_avg* h, float* loss_host) {
  if (int rc = check_bound(h)) return rc;
  DeviceScope scope(h->device);
  if (!loss_host) return HA_EINVAL;
  if (int rc = h->cuda(cudaMemcpyAsync(loss_host, h->loss(), h->P * 4, cudaMemcpyDeviceToHost,
                                       h->stream), "losses: copy"))
    return rc;
  return h->cuda(cudaStreamSynchronize(h->stream), "losses: sync");
}

int hier_avg_check(hier_avg* h) {
  if (int rc = check_bound(h)) return rc;
  DeviceScope scope(h->device);
  int word = 0;
  if (int rc = h->cuda(cudaMemcpyAsync(&word, h->err_word(), 4, cudaMemcpyDeviceToHost, h->stream),
                       "check: copy"))
    return rc;
  if (int rc = h->cuda(cudaStreamSynchronize(h->stream), "check: sync")) return rc;
  if (word) {
    cudaMemsetAsync(h->err_word(), 0, 4, h->stream);
    return h->fail(HA_ETIMEOUT, "a bounded device wait expired (error word %d)", word);
  }
  return HA_OK;
}

int hier_avg_wait_selftest(hier_avg* h, int64_t limit_us) {
  if (int rc = check_bound(h)) return rc;
  if (limit_us < 1 || limit_us > 10000000)
    return h->fail(HA_EINVAL, "wait_selftest: limit %lld us is outside [1, 1e7]",
                   (long long)limit_us);
  DeviceScope scope(h->device);
  int khz = 0;
  if (int rc = h->cuda(cudaDeviceGetAttribute(&khz, cudaDevAttrClockRate, h->device),
                       "wait_selftest: clock rate"))
    return rc;
  const long long cycles = static_cast<long long>(limit_us) * khz / 1000;
  ++h->launches;
  k_wait_selftest<<<1, 32, 0, h->stream>>>(h->never_set(), h->err_word(), cycles);
  return h->cuda(cudaGetLastError(), "wait_selftest: launch");
}

int hier_avg_launches(const hier_avg* h, int64_t* launches) {
  if (!h || !launches) return HA_EINVAL;
  *launches = h->launches;
  return HA_OK;
}

int hier_avg_profile_every(hier_avg* h, int every) {
  if (!h || every < 1) return HA_EINVAL;
  h->prof_every = every;
  return HA_OK;
}

int hier_avg_profile_kinds(hier_avg* h, unsigned kinds) {
  if (!h) return HA_EINVAL;
  if (kinds >> HA_KERNEL_KINDS) return h->fail(HA_EINVAL, "profile: unknown kernel kind bit");
  if (h->bound) cudaStreamSynchronize(h->stream);
  h->recs.clear();
  for (auto& n : h->prof_seen) n = 0;
  h->pool_used = 0;
  h->prof = kinds;
  return HA_OK;
}

int hier_avg_profile(hier_avg* h, int enable) {
  return hier_avg_profile_kinds(h, enable ? (1u << HA_KERNEL_KINDS) - 1 : 0u);
}

int hier_avg_profile_read(hier_avg* h, int kind, double* total_ms, int64_t* launches,
                          double* bytes, double* flops) {
  if (!h || kind < 0 || kind >= HA_KERNEL_KINDS) return HA_EINVAL;
  if (h->bound) {
    if (int rc = h->cuda(cudaStreamSynchronize(h->stream), "profile: sync")) return rc;
  }
  double ms = 0, by = 0, fl = 0;
  int64_t n = 0;
  for (const ProfRec& r : h->recs) {
    if (r.kind != kind) continue;
    float e = 0.f;
    if (cudaEventElapsedTime(&e, r.a, r.b) == cudaSuccess) ms += e;
    by += r.bytes;
    fl += r.flops;
    ++n;
  }
  if (total_ms) *total_ms = ms;
  if (launches) *launches = n;
  if (bytes) *bytes = by;
  if (flops) *flops = fl;
  return HA_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free step.  Some callers cannot allocate device memory at all: code
// running under an allocator they do not own, inside a host that forbids
// cudaMalloc after start-up, or from a language binding that only hands out
// existing buffers.  For them the step's scratch (activations, their transposes,
// split-K partial sums and tile counters) lives in this file-scope array instead
// of a caller workspace.  Every GPU that loads the library holds it until exit.
namespace {

constexpr int64_t kStaticScratchBytes = int64_t(32) << 20;   // 32 MiB

static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

// Unique id of the current CUDA context (ids are never reused within a process), or
// 0 if it cannot be read.
unsigned long long current_context_id() {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(p);
  });
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx ||
      get_id(ctx, &id) != CUDA_SUCCESS)
    return 0;
  return id;
}

std::mutex g_scratch_mutex;
struct ScratchAddr {
  unsigned long long ctx_id;
  void* ptr;
};
std::vector<ScratchAddr> g_scratch_addr;   // one entry per CUDA context seen

// Device address of g_static_scratch in the current context (the device must be
// current).  In host code the symbol's name is only a host-side stand-in.  The
// address is looked up once per context: a device reset creates a new context, in
// which the module (and the array) is loaded again, so an address cached for the old
// context is never reused.
cudaError_t static_scratch(void** out) {
  unsigned long long id = current_context_id();
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  if (id != 0)
    for (const ScratchAddr& a : g_scratch_addr)
      if (a.ctx_id == id) {
        *out = a.ptr;
        return cudaSuccess;
      }
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
  if (e != cudaSuccess) return e;
  if (id == 0) id = current_context_id();   // the lookup may have created the context
  if (id != 0) g_scratch_addr.push_back({id, p});
  *out = p;
  return cudaSuccess;
}

}  // namespace

extern "C" int hier_avg_step_static(hier_avg* h, float* params_dev, const void* X_dev,
                                    const int32_t* y_dev, int64_t N, void* stream) {
  if (!h) return HA_EINVAL;
  if (!params_dev || !X_dev || !y_dev || N < 1)
    return h->fail(HA_EINVAL, "step_static: NULL buffer or N < 1");
  if (h->ws_step_bytes > kStaticScratchBytes)
    return h->fail(HA_ENOMEM,
                   "step_static: this configuration needs %lld bytes of scratch, the static "
                   "array holds %lld; use hier_avg_bind with a caller workspace",
                   (long long)h->ws_step_bytes, (long long)kStaticScratchBytes);
  if (reinterpret_cast<uintptr_t>(params_dev) % 256)
    return h->fail(HA_EINVAL, "step_static: params must be 256-byte aligned");
  if (h->prec == HA_PREC_BF16 && reinterpret_cast<uintptr_t>(X_dev) % 16)
    return h->fail(HA_EINVAL, "step_static: X must be 16-byte aligned");
  cudaPointerAttributes attr;
  if (cudaPointerGetAttributes(&attr, params_dev) != cudaSuccess || attr.type != cudaMemoryTypeDevice)
    return h->fail(HA_EINVAL, "step_static: params is not device memory");
  int rc;
  DeviceScope scope(attr.device);
  int cur = -1;
  if (cudaGetDevice(&cur) != cudaSuccess || cur != attr.device)
    return h->fail(HA_ECUDA, "step_static: cannot make device %d current", attr.device);
  void* scratch = nullptr;
  if ((rc = h->cuda(static_scratch(&scratch), "step_static: scratch address"))) return rc;
  h->bound = false;
  h->device = attr.device;
  h->params = params_dev;
  h->ws = static_cast<uint8_t*>(scratch);
  h->X = X_dev;
  h->y = y_dev;
  h->N = N;
  h->stream = static_cast<cudaStream_t>(stream);
  // The array keeps whatever the previous call (of any handle) left in it; the
  // step needs its padding and its split-K counters to start at zero.
  if ((rc = h->cuda(cudaMemsetAsync(h->ws, 0, h->ws_step_bytes, h->stream), "step_static: clear")))
    return rc;
  h->m_ok = false;   // the array holds a step's scratch only: rounds average in place
  h->upd_group = 1;
  if (h->prec == HA_PREC_BF16) {
    if ((rc = h->cuda(ha::tc_configure(), "step_static: kernel attributes"))) return rc;
    if ((rc = h->cuda(ha::head_configure(), "step_static: kernel attributes"))) return rc;
    if ((rc = build_maps(h))) return rc;
  }
  h->bound = true;
  return do_step(h);
}
