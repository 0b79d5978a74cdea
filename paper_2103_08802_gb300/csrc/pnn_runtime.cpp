// Host runtime of the parareal training library: description parsing, the
// planner (values, BN norms, parameter table, forward/backward op lists per
// subnetwork), the memory plan of the single workspace, grouped launch tables,
// CUDA-graph capture, and the C ABI of include/pnn.h.
//
// Structure of one training step (Lee, Lee & Park, Algorithms 1 and 2):
//   pre wave     C^j for every j, grouped across j          (eq:xjyj, x_j)
//   fine wave    g^j for every j, grouped across j          (eq:xjyj, y_j)
//   coarse       r_j, the sequential chain F^1..F^{N-1}     (eq:correct)
//   post         h and the softmax cross-entropy loss       (eq:barf)
//   backward     post, coarse chain (D_j), fine wave, pre wave (Algorithm 2)
//   update       SGD with Nesterov momentum (Section 4)
// Ops of different subnetworks that sit at the same (block, slot) position
// are merged into one grouped launch.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <limits>
#include <map>
#include <string>
#include <tuple>
#include <vector>

#include "../../include/pnn.h"
#include "pnn_internal.h"

#include <cuda.h>
#include <cudaTypedefs.h>

using namespace pnn;

namespace {

enum Kind {
  K_CONV_FWD = 0, K_DGRAD, K_WGRAD, K_WREDUCE, K_EW, K_EW_BWD, K_BN_FIN, K_BNB_RED, K_BNB_FIN,
  K_BNB_APPLY, K_POOL_FWD, K_POOL_BWD, K_HEAD_FWD, K_HEAD_BWD, K_CONV_FWD_TC, K_DGRAD_TC, K_WGRAD_TC,
  K_NKINDS
};

struct ParamT {
  int kind;
  int dims[4];
  size_t off, n;
};

struct Value {
  int C = 0, H = 0, W = 0;
  int dt = DT_F32;
  bool virt = false;
  int src = -1, norm = -1;
  bool relu = false;
  bool need_grad = false;
  int producer = -1;  // index into ops of the producing forward op
  size_t off = 0, goff = 0;
  int galias = -1;  // gradient lives in another value's gradient buffer
  bool grad_written = false;
  int gwrites = 0;           // ops that wrote (stored or accumulated) this gradient
  int gwriter_dgrad = -1;    // the last data-gradient op among them
  // values whose gradient, times a coefficient, is to be added into this one's
  std::vector<std::pair<int, float>> pending;
};

struct Norm {
  int fused_tiles = 0;                       // BN-backward partials written by a data-gradient epilogue: its m-tiles
  int stat_rows = kEwRowsPerTile;            // rows of a forward-statistics partial tile
  int C = 0, h = -1, gamma = -1, beta = -1;  // gamma/beta: param ids
  int virt = -1;                             // the virtual BN(+ReLU) value
  int tiles = 0;
  int64_t count = 0;
  size_t part = 0, mean = 0, rstd = 0, scale = 0, shift = 0, bpart = 0, coef = 0;
  int btiles = 0;
  size_t run = 0;  // running mean (C floats) followed by running variance (C floats)
  // finalize reductions (forward statistics, backward sums): chunk scratch and
  // per-channel-group counters
  size_t fscr = 0, fcnt = 0, bscr = 0, bcnt = 0;
};

// One planned op (forward or backward).  Fields are interpreted per kind.
struct POp {
  int kind = 0;
  int variant = 0;
  int key[3] = {0, 0, 0};
  int in = -1, out = -1, res = -1, w = -1;   // conv: values / param id
  int k = 1, stride = 1, pad = 0;
  int stats_norm = -1;
  int ins[3] = {-1, -1, -1};
  float coef[3] = {0, 0, 0};
  int nin = 0;
  bool relu = false;
  int norm = -1;
  int acc = 0;                               // accumulate into the written gradient
  int acc_in[3] = {0, 0, 0};
  int addv[2] = {-1, -1};                    // BNB_APPLY: extra gradients added into dh
  float addc[2] = {1.f, 1.f};                // ... with these coefficients
  int res2[2] = {-1, -1};                    // conv forward: more addends of the output
  float rcoef[2] = {0.f, 0.f};               // ... with these coefficients
  int splits = 1, pix_per_split = 0;
  int bn_fuse = -1;                          // TMA dgrad: norm whose BN-backward partials the epilogue writes
  size_t scratch = 0;                        // wgrad partial buffer offset
  int tiles = 0, mtiles = 0, ntiles = 0;
  int head = 0;
};

struct Launch {
  int kind, variant;
  size_t table_off, tstart_off;
  int count, total;
  int phase;
  int aux;  // tcgen05 conv: largest N tile of the group
  double flops, bytes;  // algorithmic work of this launch
  int shape[6];         // first op: conv (C_in, C_out, k, stride, H_out, W_out); else (C, H, W, 0, 0, 0)
  int esz = 4;          // TMA-fed conv: largest element size of the A sources
  int raw = 0;          // TMA-fed conv: raw slot bytes of one stage
  int op = 0;           // TMA-fed conv with halo tiles: operand slot bytes of one stage (0: default)
  int wide = 0;         // TMA-fed forward / data gradient: every tile one k-step (the wide-epilogue variant)
  int block = -1;       // fine forward / backward: position of the layer in its segment
};

// Tile and kernel-choice rules shared with the single-convolution entry
// points (pnn_internal.h), in terms of this file's kinds.
static int conv_mode(int kind) { return kind == K_DGRAD_TC ? 1 : (kind == K_WGRAD_TC ? 2 : 0); }
static int tc_ntile_w(int kind, int variant) { return tc_ntile_cols(conv_mode(kind), variant); }
static int tc_mtile_rows(int kind, int variant, int C) { return tc_tile_rows(conv_mode(kind), variant, C); }
// conv_impl values with the TMA-fed kernels (4: without halo tiles)
static bool tma_impl(int conv_impl) { return conv_impl == 0 || conv_impl == 4; }
// a TMA-fed 3x3 forward / data gradient instance that takes halo tiles:
// A source H x W x ch, N tile bn
static bool use_halo(int conv_impl, int mode, int k, int stride, int pad, int H, int W, int ch, int bn) {
  return conv_impl == 0 && halo_ok(k, stride, pad, H, W, ch) && conv_halo_fits(mode, W, ch, bn);
}
static int tma_bn(int mode, int ncols) {
  return ncols <= tc_ntile_cols(mode, 1) ? ((ncols + 15) & ~15) : tc_ntile_cols(mode, 1);
}

const char* kKindName[K_NKINDS] = {"conv_fwd", "conv_dgrad", "conv_wgrad", "wgrad_reduce", "elementwise",
                                   "elementwise_bwd", "bn_finalize", "bn_bwd_reduce", "bn_bwd_finalize",
                                   "bn_bwd_apply", "pool_fwd", "pool_bwd", "head_fwd", "head_bwd",
                                   "conv_fwd_tc", "conv_dgrad_tc", "conv_wgrad_tc"};

struct Phase { std::vector<Launch> launches; };

int cdiv(int64_t a, int64_t b) { return (int)((a + b - 1) / b); }
size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

struct Group {
  int kind, variant;
  std::vector<int> ops;
};

}  // namespace

struct pnn_net {
  // description
  int B = 0, in_c = 0, in_h = 0, in_w = 0, classes = 0, N = 0;
  int head_kind = 0;
  std::vector<int> head_hidden;
  pnn_options opt{};
  int act_dt = DT_BF16, stream_dt = DT_F32;
  bool use_tc = false;
  // plan
  std::vector<ParamT> params;
  size_t nparams = 0;
  std::vector<Value> vals;
  std::vector<Norm> norms;
  std::vector<POp> ops;  // all planned ops
  // op-index sequences
  std::vector<std::vector<int>> pre_f, fine_f, delta_f, pre_b, fine_b, delta_b;
  std::vector<int> coarse_f, head_f, coarse_b, head_b;
  // interface values
  int x_in = -1;
  std::vector<int> xs, ys, rs, rts;
  int ytilde = -1;
  // the correction folded into conv epilogues: y_j (j < N) not stored (the
  // value ys[j] holds r_j = y_j - x_{j+1}), rt_N not stored (rts[N-1] is
  // ytilde = y_N + rt_N)
  std::vector<char> y_is_r;
  bool rtN_in_ytilde = false;
  // interface tensors the step does not store, exported as a + c * b of two
  // stored values: (which, j) -> (a, b, c)
  std::map<std::pair<int, int>, std::tuple<int, int, float>> derived;
  // head
  int head_in = -1, head_norm = -1;
  std::vector<int> fc_w, fc_b;
  std::vector<int> fc_width;
  size_t feat_off = 0;                 // [nfc+1] feature buffers
  std::vector<size_t> feat, dfeat;
  size_t logits_off = 0, dlogits_off = 0, loss_off = 0, status_off = 0;
  size_t labels_stage = 0, x_stage = 0, export_off = 0;
  size_t export_bytes = 0;
  // memory
  size_t off_master = 0, off_grad = 0, off_mom = 0, off_shadow = 0, off_wt = 0;
  // weight transpose launch (bf16 mode): Wt[c][r][s][k] for the tensor-core data gradient
  size_t wt_tab = 0, wt_ts = 0;
  int wt_count = 0, wt_total = 0;
  size_t ws_bytes = 0, cursor = 0;
  size_t tables_off = 0, tables_bytes = 0;
  char* ws = nullptr;
  // launch lists
  // 0 pre_f 1 fine_f(+delta_f) 2 coarse_f 3 head_f 4 head_b 5 coarse_b 6 delta_b 7 fine_b 8 pre_b
  Phase ph[11];  // 0-8 the step's phases; 9 the last subnetwork's backward and 10 the
                 // deferred x_N gradient term when the coarse chain overlaps it
  std::vector<uint8_t> host_tables;
  std::vector<size_t> run_at;   // param id of a BN gamma -> float offset of its running statistics
  // coarse/fine overlap: the last subnetwork's backward (it needs only D_N) runs
  // on s_lo beside the coarse chain's backward on s_hi; the chain's term
  // -dL/dr_{N-1} of dL/dx_N is deferred to fix_b, after both
  bool overlap_on = false;
  int defer_x = -1, defer_r = -1;
  std::vector<int> fix_b;
  cudaStream_t s_hi = nullptr, s_lo = nullptr;
  cudaEvent_t fork_ev = nullptr, hi_done = nullptr, lo_done = nullptr;
  int lo_cap = 0;  // grid cap of s_lo's persistent kernels
  size_t running_floats = 0, off_running = 0;
  size_t off_fin_cnt = 0, fin_cnt_bytes = 0;
  // pnn_infer's graph, captured for (ix, ilogits)
  cudaGraphExec_t igexec = nullptr;
  const float* ix = nullptr;
  float* ilogits = nullptr;
  // runtime state
  cudaStream_t stream = nullptr;
  bool own_stream = false;
  int state = 0;  // 0 idle, 1 forward done, 2 backward done
  bool first_step = true;
  const float* x_dev = nullptr;
  const int32_t* labels_dev = nullptr;
  float* loss_dev = nullptr;
  cudaEvent_t ev[12] = {};
  bool events = false;
  float timings[10] = {};
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t gexec = nullptr;
  const float* g_x = nullptr;
  const int32_t* g_labels = nullptr;
  float* g_loss = nullptr;
  // one graph per phase for pnn_time_phases (pre, fine, coarse, post forward;
  // post, coarse, fine, pre backward; update), captured for (px, plabels)
  cudaGraphExec_t pgexec[9] = {};
  const float* px = nullptr;
  const int32_t* plabels = nullptr;
  std::string err;
  int counts[3] = {0, 0, 0};
  // profiling: events around every launch, accumulated per kind
  bool prof = false;
  std::vector<cudaEvent_t> pev;
  std::vector<const Launch*> plaunch;
  size_t pnext = 0, pfold = 0;
  double kms[K_NKINDS + 1] = {}, kflops[K_NKINDS + 1] = {}, kbytes[K_NKINDS + 1] = {};
  int64_t klaunch[K_NKINDS + 1] = {};

  template <class T> T* P(size_t off) const { return reinterpret_cast<T*>(ws + off); }

  // ------------------------------------------------------------ planning
  size_t alloc(size_t bytes) {
    size_t o = cursor;
    cursor = align256(cursor + bytes);
    return o;
  }
  int add_param(int kind, int d0, int d1 = 1, int d2 = 1, int d3 = 1) {
    ParamT p;
    p.kind = kind;
    p.dims[0] = d0; p.dims[1] = d1; p.dims[2] = d2; p.dims[3] = d3;
    p.off = nparams;
    p.n = (size_t)d0 * d1 * d2 * d3;
    nparams += p.n;
    params.push_back(p);
    return (int)params.size() - 1;
  }
  int new_value(int C, int H, int W, int dt, bool need_grad) {
    Value v;
    v.C = C; v.H = H; v.W = W; v.dt = dt; v.need_grad = need_grad;
    vals.push_back(v);
    return (int)vals.size() - 1;
  }
  int64_t rows(int v) const { return (int64_t)B * vals[v].H * vals[v].W; }
  int new_op(std::vector<int>& list, const POp& op) {
    ops.push_back(op);
    list.push_back((int)ops.size() - 1);
    return (int)ops.size() - 1;
  }
  // Make sure BN partial statistics of value h are produced; returns tiles.
  void request_stats(std::vector<int>& list, int nid, int h, int key0) {
    Value& hv = vals[h];
    if (hv.producer >= 0) {
      POp& p = ops[hv.producer];
      if ((p.kind == K_CONV_FWD || p.kind == K_CONV_FWD_TC || (p.kind == K_EW && p.out == h)) && p.stats_norm < 0) {
        p.stats_norm = nid;
        norms[nid].tiles = p.tiles;
        norms[nid].stat_rows = p.kind == K_CONV_FWD_TC ? kTcBM
                               : p.kind == K_CONV_FWD  ? simt_tile(p.variant).BM
                                                       : kEwRowsPerTile;
        return;
      }
    }
    POp s;
    s.kind = K_EW;
    s.ins[0] = h; s.coef[0] = 1.f; s.nin = 1; s.out = -1;
    s.stats_norm = nid;
    s.tiles = cdiv(rows(h), kEwRowsPerTile);
    s.key[0] = key0; s.key[1] = 90;
    norms[nid].tiles = s.tiles;
    norms[nid].stat_rows = kEwRowsPerTile;
    new_op(list, s);
  }
  // virtual BN(+ReLU) of h with fresh or given gamma/beta params
  int bn_virtual(std::vector<int>& list, int h, int gamma, int beta, bool relu, int key0, int slot) {
    Norm n;
    n.C = vals[h].C; n.h = h; n.gamma = gamma; n.beta = beta;
    n.count = rows(h);
    norms.push_back(n);
    int nid = (int)norms.size() - 1;
    if (!opt.inference) request_stats(list, nid, h, key0);  // inference normalises with running statistics
    POp f;
    f.kind = K_BN_FIN; f.norm = nid;
    f.key[0] = key0; f.key[1] = slot;
    new_op(list, f);
    Value v;
    v.C = vals[h].C; v.H = vals[h].H; v.W = vals[h].W; v.dt = DT_F32;
    v.virt = true; v.src = h; v.norm = nid; v.relu = relu; v.need_grad = true;
    vals.push_back(v);
    norms[nid].virt = (int)vals.size() - 1;
    return (int)vals.size() - 1;
  }
  int conv(std::vector<int>& list, int in, int w, int cout, int k, int stride, int res, int out_dt, int key0,
           int slot) {
    const Value iv = vals[in];  // a copy: new_value() below may reallocate vals
    int P = (iv.H + 2 * (k / 2) - k) / stride + 1, Q = (iv.W + 2 * (k / 2) - k) / stride + 1;
    int out = new_value(cout, P, Q, out_dt, true);
    POp c;
    c.kind = K_CONV_FWD;
    c.in = in; c.out = out; c.res = res; c.w = w; c.k = k; c.stride = stride; c.pad = k / 2;
    c.key[0] = key0; c.key[1] = slot;
    int M = B * P * Q;
    if (act_dt == DT_BF16 && (tma_impl(opt.conv_impl) || opt.conv_impl == 3) && iv.C % 8 == 0 && cout % 8 == 0) {
      // tcgen05 path: 128-pixel tiles, all output channels (<= 256) per tile
      c.kind = K_CONV_FWD_TC;
      // the TMA-fed forward (eight epilogue warps) pays off when the epilogue
      // is wide (measured: 2x on 16->64 with the residual) or when the 3x3
      // taps come from one halo box; other narrow outputs keep the
      // thread-gathered kernel, which is faster there
      const bool halo = use_halo(opt.conv_impl, 0, k, stride, k / 2, iv.H, iv.W, iv.C, tma_bn(0, cout));
      c.variant = tma_impl(opt.conv_impl) && ((cout >= 64 && tma_shape_ok(k, stride, k / 2, iv.C)) || halo) ? 1 : 0;
      c.mtiles = cdiv(M, kTcBM);
      c.ntiles = cdiv(cout, tc_ntile_w(c.kind, c.variant));
    } else {
      c.variant = cout <= 16 ? 2 : (cout <= 32 ? 1 : 0);
      ConvTile t = simt_tile(c.variant);
      c.mtiles = cdiv(M, t.BM);
      c.ntiles = cdiv(cout, t.BN);
    }
    c.tiles = c.mtiles;  // stats partial rows
    int id = new_op(list, c);
    vals[out].producer = id;
    return out;
  }
  int ew(std::vector<int>& list, std::vector<int> ins, std::vector<float> coef, bool relu, int out_dt, int key0,
         int slot) {
    const Value a = vals[ins[0]];  // a copy: new_value() below may reallocate vals
    bool ng = false;
    for (int i : ins) ng = ng || vals[i].need_grad;
    int out = new_value(a.C, a.H, a.W, out_dt, ng);
    POp e;
    e.kind = K_EW;
    e.nin = (int)ins.size();
    for (int i = 0; i < e.nin; ++i) { e.ins[i] = ins[i]; e.coef[i] = coef[i]; }
    e.out = out; e.relu = relu;
    e.tiles = cdiv(rows(out), kEwRowsPerTile);
    e.key[0] = key0; e.key[1] = slot;
    int id = new_op(list, e);
    vals[out].producer = id;
    return out;
  }
  int pool(std::vector<int>& list, int in, int k, int s, int p, int key0, int slot) {
    const Value iv = vals[in];  // a copy: new_value() below may reallocate vals
    int P = (iv.H + 2 * p - k) / s + 1, Q = (iv.W + 2 * p - k) / s + 1;
    int out = new_value(iv.C, P, Q, iv.virt ? act_dt : iv.dt, iv.need_grad);
    POp o;
    o.kind = K_POOL_FWD; o.in = in; o.out = out; o.k = k; o.stride = s; o.pad = p;
    o.tiles = cdiv((int64_t)B * P * Q * iv.C, 256);
    o.key[0] = key0; o.key[1] = slot;
    int id = new_op(list, o);
    vals[out].producer = id;
    return out;
  }

  // A parameter cursor lets the delta correction evaluate F^j twice with one
  // set of parameters.
  struct PCur {
    std::vector<int>* ids;
    size_t i;
    bool replay;
  };
  int take(PCur& pc, int kind, int d0, int d1 = 1, int d2 = 1, int d3 = 1) {
    if (pc.replay) return (*pc.ids)[pc.i++];
    int id = add_param(kind, d0, d1, d2, d3);
    pc.ids->push_back(id);
    return id;
  }

  // one layer of the description; returns its output value
  int layer(std::vector<int>& L, const pnn_layer& ly, int x, PCur& pc, int key0, bool resid_stream) {
    const int cin = vals[x].C;
    const int sdt = resid_stream ? stream_dt : act_dt;
    switch (ly.op) {
      case PNN_CONV: {
        int w = take(pc, 0, ly.cout, cin, ly.k, ly.k);
        return conv(L, x, w, ly.cout, ly.k, ly.stride, -1, act_dt, key0, 0);
      }
      case PNN_CONV_BN_RELU: {
        int w = take(pc, 0, ly.cout, cin, ly.k, ly.k);
        int g = take(pc, 1, ly.cout), b = take(pc, 2, ly.cout);
        int h = conv(L, x, w, ly.cout, ly.k, ly.stride, -1, act_dt, key0, 0);
        int a = bn_virtual(L, h, g, b, true, key0, 1);
        if (ly.pool) return pool(L, a, 2, 2, 0, key0, 2);
        return a;
      }
      case PNN_BASIC: {
        int w1 = take(pc, 0, ly.cout, cin, 3, 3);
        int g1 = take(pc, 1, ly.cout), b1 = take(pc, 2, ly.cout);
        int w2 = take(pc, 0, ly.cout, ly.cout, 3, 3);
        int g2 = take(pc, 1, ly.cout), b2 = take(pc, 2, ly.cout);
        int h1 = conv(L, x, w1, ly.cout, 3, 1, -1, act_dt, key0, 0);
        int a1 = bn_virtual(L, h1, g1, b1, true, key0, 1);
        int h2 = conv(L, a1, w2, ly.cout, 3, 1, -1, act_dt, key0, 2);
        int z2 = bn_virtual(L, h2, g2, b2, false, key0, 3);
        return ew(L, {z2, x}, {1.f, 1.f}, true, sdt, key0, 4);
      }
      case PNN_BOTTLENECK: {
        const bool proj = cin != ly.cout || ly.stride != 1;
        int g1 = take(pc, 1, cin), b1 = take(pc, 2, cin);
        int w1 = take(pc, 0, ly.mid, cin, 1, 1);
        int g2 = take(pc, 1, ly.mid), b2 = take(pc, 2, ly.mid);
        int w2 = take(pc, 0, ly.mid, ly.mid, 3, 3);
        int g3 = take(pc, 1, ly.mid), b3 = take(pc, 2, ly.mid);
        int w3 = take(pc, 0, ly.cout, ly.mid, 1, 1);
        int wp = proj ? take(pc, 0, ly.cout, cin, 1, 1) : -1;
        int a1 = bn_virtual(L, x, g1, b1, true, key0, 0);
        int h1 = conv(L, a1, w1, ly.mid, 1, 1, -1, act_dt, key0, 1);
        int a2 = bn_virtual(L, h1, g2, b2, true, key0, 2);
        int h2 = conv(L, a2, w2, ly.mid, 3, ly.stride, -1, act_dt, key0, 3);
        int a3 = bn_virtual(L, h2, g3, b3, true, key0, 4);
        int sc = proj ? conv(L, a1, wp, ly.cout, 1, ly.stride, -1, act_dt, key0, 5) : x;
        if (vals[sc].virt) sc = ew(L, {sc}, {1.f}, false, sdt, key0, 5);
        return conv(L, a3, w3, ly.cout, 1, 1, sc, sdt, key0, 6);
      }
      case PNN_COARSE_RU: {
        const bool proj = cin != ly.cout || ly.stride != 1;
        int g1 = take(pc, 1, cin), b1 = take(pc, 2, cin);
        int w1 = take(pc, 0, ly.cout, cin, 3, 3);
        int g2 = take(pc, 1, ly.cout), b2 = take(pc, 2, ly.cout);
        int w2 = take(pc, 0, ly.cout, ly.cout, 3, 3);
        int wp = proj ? take(pc, 0, ly.cout, cin, 1, 1) : -1;
        int a1 = bn_virtual(L, x, g1, b1, true, key0, 0);
        int h1 = conv(L, a1, w1, ly.cout, 3, ly.stride, -1, act_dt, key0, 1);
        int a2 = bn_virtual(L, h1, g2, b2, true, key0, 2);
        int sc = proj ? conv(L, a1, wp, ly.cout, 1, ly.stride, -1, act_dt, key0, 3) : x;
        if (vals[sc].virt) sc = ew(L, {sc}, {1.f}, false, sdt, key0, 3);
        return conv(L, a2, w2, ly.cout, 3, 1, sc, sdt, key0, 4);
      }
    }
    return -1;
  }
  int stack(std::vector<int>& L, const pnn_layer* ls, int n, int x, PCur& pc, int key_base, bool resid_stream) {
    for (int i = 0; i < n; ++i) x = layer(L, ls[i], x, pc, key_base + i, resid_stream);
    return x;
  }

  // ------------------------------------------------------------ backward planning
  int grad_acc(int v) {
    int a = vals[v].grad_written ? 1 : 0;
    vals[v].grad_written = true;
    vals[v].gwrites++;
    return a;
  }
  void flush_pending(std::vector<int>& L, int v, const int* key) {
    // add pending residual gradients of v as plain accumulate ops
    for (const auto& pc : vals[v].pending) {
      const int src = pc.first;
      POp e;
      e.kind = K_EW_BWD;
      e.in = src;  // dout = grad(src)
      e.out = -1;
      e.nin = 1; e.ins[0] = v; e.coef[0] = pc.second; e.acc_in[0] = grad_acc(v);
      e.tiles = cdiv(rows(v), kEwRowsPerTile);
      e.key[0] = key[0]; e.key[1] = key[1]; e.key[2] = 9;
      new_op(L, e);
    }
    vals[v].pending.clear();
  }
  // Before a gradient is read it must be complete: residual contributions
  // still pending become an alias (single source, nothing else written) or
  // explicit accumulate ops.
  void resolve(std::vector<int>& L, int v, const int* key) {
    Value& x = vals[v];
    if (x.pending.empty()) return;
    if (!x.grad_written && x.pending.size() == 1 && x.pending[0].second == 1.f) {
      x.galias = x.pending[0].first;
      x.grad_written = true;
      x.pending.clear();
      return;
    }
    flush_pending(L, v, key);
  }
  size_t gptr(int v) const {
    while (vals[v].galias >= 0) v = vals[v].galias;
    return vals[v].goff;
  }
  void backward_of(std::vector<int>& L, int fid) {
    const POp f = ops[fid];
    const int k0 = -f.key[0], k1 = -f.key[1];
    {
      const int key_[2] = {k0, k1};
      if (f.out >= 0) resolve(L, f.out, key_);
      if (f.kind == K_BN_FIN && norms[f.norm].virt >= 0) resolve(L, norms[f.norm].virt, key_);
    }
    auto key = [&](POp& o, int sub) { o.key[0] = k0; o.key[1] = k1; o.key[2] = sub; };
    switch (f.kind) {
      case K_CONV_FWD:
      case K_CONV_FWD_TC: {
        const Value& ov = vals[f.out];
        if (f.res >= 0 && vals[f.res].need_grad) vals[f.res].pending.push_back({f.out, 1.f});
        for (int e = 0; e < 2; ++e)
          if (f.res2[e] >= 0 && vals[f.res2[e]].need_grad) vals[f.res2[e]].pending.push_back({f.out, f.rcoef[e]});
        POp wg;
        wg.kind = K_WGRAD; wg.in = f.in; wg.out = f.out; wg.w = f.w; wg.k = f.k; wg.stride = f.stride; wg.pad = f.pad;
        const int RSC = f.k * f.k * vals[f.in].C;
        const int64_t Mp = (int64_t)B * ov.H * ov.W;
        const bool tc_ok = act_dt == DT_BF16 && opt.conv_impl != 1 && vals[f.in].C % 8 == 0 && ov.C % 8 == 0;
        int pix_align = kWgradBK;
        if (tc_ok) {
          // tensor cores: rows (r,s,c) in 128-row tiles, all k_out per tile, pixels split across CTAs
          wg.kind = K_WGRAD_TC;
          {
            const int src = vals[f.in].virt ? vals[f.in].src : f.in;
            wg.variant = tma_impl(opt.conv_impl) && tma_wgrad_ok(f.k, f.stride, f.pad, vals[f.in].C, ov.C, vals[f.in].W,
                                                             vals[src].dt == DT_BF16)
                             ? 1
                             : 0;
          }
          wg.mtiles = cdiv(RSC, tc_mtile_rows(wg.kind, wg.variant, vals[f.in].C));
          wg.ntiles = cdiv(ov.C, 256);
          pix_align = 64;
        } else {
          wg.mtiles = cdiv(ov.C, kWgradBM);
          wg.ntiles = cdiv(RSC, kWgradBN);
          // few input channels (the 3-channel stem and C^j convs): the
          // kernel that stages the im2col operand once per pixel step
          wg.variant = vals[f.in].C < 8 && RSC <= kWgradBN ? 1 : 0;
        }
        int base = wg.mtiles * wg.ntiles;
        int splits = std::max(1, std::min(cdiv(Mp, 256), cdiv(2 * (int64_t)device_sm_count(), base)));
        wg.pix_per_split = cdiv(cdiv(Mp, splits), pix_align) * pix_align;
        wg.splits = cdiv(Mp, wg.pix_per_split);
        wg.tiles = base * wg.splits;
        key(wg, 0);
        new_op(L, wg);
        POp rd;
        rd.kind = K_WREDUCE; rd.w = f.w; rd.splits = wg.splits; rd.out = f.out; rd.in = f.in; rd.k = f.k;
        rd.variant = tc_ok ? 1 : 0;  // partial layout of the matching wgrad
        rd.tiles = cdiv((int64_t)ov.C * RSC, 32);  // 32 elements per CTA
        key(rd, 1);
        new_op(L, rd);
        if (vals[f.in].need_grad) {
          flush_pending(L, f.in, rd.key);
          POp dg;
          dg.kind = K_DGRAD; dg.in = f.in; dg.out = f.out; dg.w = f.w; dg.k = f.k; dg.stride = f.stride; dg.pad = f.pad;
          const Value& iv = vals[f.in];
          if (act_dt == DT_BF16 && opt.conv_impl != 1 && iv.C % 8 == 0 && ov.C % 8 == 0 && params[f.w].off % 8 == 0) {
            dg.kind = K_DGRAD_TC;
            const int bn = tma_bn(1, iv.C);
            dg.variant = tma_impl(opt.conv_impl) && (tma_shape_ok(f.k, f.stride, f.pad, ov.C) ||
                                                     use_halo(opt.conv_impl, 1, f.k, f.stride, f.pad, ov.H, ov.W, ov.C, bn))
                             ? 1
                             : 0;
            dg.mtiles = cdiv((int64_t)B * iv.H * iv.W, kTcBM);
            dg.ntiles = cdiv(iv.C, tc_ntile_w(dg.kind, dg.variant));
          } else {
            dg.variant = iv.C <= 16 ? 2 : (iv.C <= 32 ? 1 : 0);
            ConvTile t = simt_tile(dg.variant);
            dg.mtiles = cdiv((int64_t)B * iv.H * iv.W, t.BM);
            dg.ntiles = cdiv(iv.C, t.BN);
          }
          dg.tiles = dg.mtiles * dg.ntiles;
          dg.acc = grad_acc(f.in);
          key(dg, 2);
          vals[f.in].gwriter_dgrad = new_op(L, dg);
        }
        break;
      }
      case K_EW: {
        if (f.out < 0) break;  // statistics only
        POp e;
        e.kind = K_EW_BWD;
        e.in = f.out; e.out = f.out; e.relu = f.relu;
        for (int i = 0; i < f.nin; ++i) {
          if (!vals[f.ins[i]].need_grad) continue;
          if (overlap_on && f.out == defer_r && f.ins[i] == defer_x) continue;  // planned into fix_b
          const int key_[2] = {k0, k1};
          flush_pending(L, f.ins[i], key_);
          e.ins[e.nin] = f.ins[i];
          e.coef[e.nin] = f.coef[i];
          e.acc_in[e.nin] = grad_acc(f.ins[i]);
          e.nin++;
        }
        if (e.nin == 0) break;
        e.tiles = cdiv(rows(f.out), kEwRowsPerTile);
        key(e, 0);
        new_op(L, e);
        break;
      }
      case K_POOL_FWD: {
        if (!vals[f.in].need_grad) break;
        const int key_[2] = {k0, k1};
        flush_pending(L, f.in, key_);
        POp p;
        p.kind = K_POOL_BWD; p.in = f.in; p.out = f.out; p.k = f.k; p.stride = f.stride; p.pad = f.pad;
        p.acc = grad_acc(f.in);
        p.tiles = cdiv(rows(f.in) * vals[f.in].C, 256);
        key(p, 0);
        new_op(L, p);
        break;
      }
      case K_BN_FIN: {
        // the virtual value of this norm has received all its gradient
        const Norm& n = norms[f.norm];
        const int vv = n.virt;
        if (vv < 0 || !vals[vv].grad_written) break;
        POp r;
        r.kind = K_BNB_RED; r.norm = f.norm; r.in = vv;
        r.variant = (n.C % 8 == 0 && n.C <= 2048) ? 1 : 0;  // 1: 8 channels per thread
        r.tiles = cdiv(n.count, bnb_rows_per_tile(n.C));
        key(r, 0);
        // The reduction is fused into the data gradient that wrote the whole
        // gradient of the BN(+ReLU) value (TMA-fed, stored, sole writer): its
        // epilogue writes the partial sums of each 128-row tile.
        const int wr = vals[vv].gwriter_dgrad;
        const bool fuse = vals[vv].gwrites == 1 && wr >= 0 && ops[wr].kind == K_DGRAD_TC && ops[wr].variant == 1 &&
                          ops[wr].acc == 0 &&
                          ops[wr].in == vv && vals[vv].galias < 0 && vals[vv].pending.empty() && n.C % 16 == 0;
        if (fuse) {
          ops[wr].bn_fuse = f.norm;
          norms[f.norm].fused_tiles = ops[wr].mtiles;
        } else {
          new_op(L, r);
        }
        POp fi = r;
        fi.kind = K_BNB_FIN;
        fi.tiles = n.C;  // one CTA per channel
        key(fi, 1);
        new_op(L, fi);
        POp ap = r;
        ap.kind = K_BNB_APPLY;
        ap.tiles = cdiv(n.count, bnb_rows_per_tile(n.C));
        if (vals[n.h].need_grad) {
          ap.acc = grad_acc(n.h);
          ap.out = n.h;
          key(ap, 2);
          // residual gradients pending on h are folded into this apply
          for (int i = 0; i < 2 && !vals[n.h].pending.empty(); ++i) {
            ap.addv[i] = vals[n.h].pending.back().first;
            ap.addc[i] = vals[n.h].pending.back().second;
            vals[n.h].pending.pop_back();
          }
          new_op(L, ap);
          const int key_[2] = {k0, k1};
          flush_pending(L, n.h, key_);
        }
        break;
      }
      case K_HEAD_FWD: {
        POp h;
        h.kind = K_HEAD_BWD;
        h.in = f.in;
        h.acc = grad_acc(f.in);
        key(h, 0);
        new_op(L, h);
        break;
      }
      default:
        break;
    }
  }
  void backward_list(const std::vector<int>& fwd, std::vector<int>& bwd) {
    for (int i = (int)fwd.size() - 1; i >= 0; --i) backward_of(bwd, fwd[i]);
  }

  // 2-D tensor map over rows x inner elements (row pitch inner * element
  // size) with box [box_rows][box_inner]; swz: swizzle span in bytes (128: the
  // MMA's K-major operand layout; 64 / 32: epilogue staging tiles; 0: dense
  // rows).  Loads read zeros outside the tensor; stores skip it.
  int encode_map(CUtensorMap* m, const void* base, bool bf16, int64_t inner, int64_t rows, int box_inner,
                 int box_rows, int swz) {
    const char* why = nullptr;
    if (encode_tensor_map_2d(m, base, bf16, inner, rows, box_inner, box_rows, swz, &why) != 0)
      return fail(PNN_ECUDA, why);
    return PNN_OK;
  }
  size_t put_table(const void* p, size_t n) {
    size_t o = align256(host_tables.size());
    host_tables.resize(o + n);
    memcpy(host_tables.data() + o, p, n);
    return o;
  }
  // head GEMM tables: per FC layer l: forward, dW, dIn descriptors
  std::vector<size_t> head_fwd_tab, head_dw_tab, head_din_tab;
  size_t head_tstart = 0;
  void build_head_tables();
  int run_head_fwd();
  int run_head_bwd(int opid);
  int plan(const pnn_desc* d);
  int bind(void* dev, size_t bytes);
  int build_tables();
  std::vector<Group> phase_groups(int p) const;
  // Inference plan: a value's buffer is handed to a later value of the same
  // size once the last launch that reads it has been issued.
  void share_activation_buffers() {
    std::vector<int> def(vals.size(), -1), last(vals.size(), -1);
    auto reads = [&](int v, int at) {
      if (v < 0) return;
      if (vals[v].virt) v = vals[v].src;
      last[v] = std::max(last[v], at);
    };
    int li = 0;
    for (int p = 0; p < 4; ++p)
      for (const Group& g : phase_groups(p)) {
        for (int id : g.ops) {
          const POp& o = ops[id];
          reads(o.in, li);
          reads(o.res, li);
          reads(o.res2[0], li);
          reads(o.res2[1], li);
          for (int i = 0; i < o.nin; ++i) reads(o.ins[i], li);
          if (o.out >= 0 && !vals[o.out].virt && def[o.out] < 0) def[o.out] = li;
        }
        ++li;
      }
    std::vector<std::vector<int>> born(li + 1), dies(li + 1);
    for (size_t v = 0; v < vals.size(); ++v) {
      if (vals[v].virt) continue;
      const int d = std::max(def[v], 0);  // the packed input is written before launch 0
      born[d].push_back((int)v);
      dies[std::max(last[v], d)].push_back((int)v);
    }
    auto bytes = [&](int v) {
      const Value& x = vals[v];
      return align256((size_t)B * x.H * x.W * x.C * (x.dt == DT_F32 ? 4 : 2));
    };
    std::map<size_t, std::vector<size_t>> free_at;  // size -> free offsets
    for (int t = 0; t <= li; ++t) {
      for (int v : born[t]) {
        std::vector<size_t>& f = free_at[bytes(v)];
        if (f.empty()) {
          vals[v].off = alloc(bytes(v));
        } else {
          vals[v].off = f.back();
          f.pop_back();
        }
      }
      for (int v : dies[t]) free_at[bytes(v)].push_back(vals[v].off);
    }
  }
  // Algorithmic work of one op, added to flops / bytes: conv FLOPs =
  // 2 * B*P*Q*K*C*R*S; bytes = each operand read once, each result written once
  // (a read-modify-write for accumulating results).
  void op_cost(const POp& o, double& flops, double& bytes) const {
    auto esz = [&](int v) {
      return vals[v].virt ? (vals[vals[v].src].dt == DT_F32 ? 4.0 : 2.0) : (vals[v].dt == DT_F32 ? 4.0 : 2.0);
    };
    auto elems = [&](int v) { return (double)B * vals[v].H * vals[v].W * vals[v].C; };
    const double wsz = act_dt == DT_BF16 ? 2.0 : 4.0;
    switch (o.kind) {
      case K_CONV_FWD: case K_CONV_FWD_TC: case K_DGRAD: case K_DGRAD_TC: case K_WGRAD: case K_WGRAD_TC: {
        const Value& iv = vals[o.in]; const Value& ov = vals[o.out];
        const double macs = (double)B * ov.H * ov.W * ov.C * iv.C * o.k * o.k;
        flops += 2 * macs;
        const double wbytes = (double)ov.C * iv.C * o.k * o.k * wsz;
        if (o.kind == K_CONV_FWD || o.kind == K_CONV_FWD_TC)
          bytes += elems(o.in) * esz(o.in) + wbytes + elems(o.out) * esz(o.out) + (o.res >= 0 ? elems(o.res) * esz(o.res) : 0) +
                   (o.res2[0] >= 0 ? elems(o.res2[0]) * esz(o.res2[0]) : 0) +
                   (o.res2[1] >= 0 ? elems(o.res2[1]) * esz(o.res2[1]) : 0);
        else if (o.kind == K_DGRAD || o.kind == K_DGRAD_TC)
          bytes += elems(o.out) * 4 + wbytes + elems(o.in) * 4 * (o.acc ? 2 : 1);
        else
          bytes += elems(o.in) * esz(o.in) + elems(o.out) * 4 + (double)o.splits * ov.C * iv.C * o.k * o.k * 4;
        break;
      }
      case K_EW: {
        const int ref = o.out >= 0 ? o.out : o.ins[0];
        for (int i = 0; i < o.nin; ++i) bytes += elems(o.ins[i]) * esz(o.ins[i]);
        if (o.out >= 0) bytes += elems(ref) * esz(ref);
        break;
      }
      case K_EW_BWD: bytes += elems(o.in) * 4 * (1 + o.nin) + (o.relu ? elems(o.in) * esz(o.in) : 0); break;
      case K_BNB_RED: bytes += elems(o.in) * 4 + elems(norms[o.norm].h) * esz(norms[o.norm].h); break;
      case K_BNB_APPLY:
        bytes += elems(o.in) * 4 + elems(norms[o.norm].h) * esz(norms[o.norm].h) + elems(norms[o.norm].h) * 4 * (o.acc ? 2 : 1);
        break;
      case K_POOL_FWD: bytes += elems(o.in) * esz(o.in) + elems(o.out) * esz(o.out); break;
      case K_POOL_BWD: bytes += elems(o.out) * 4 + elems(o.in) * (esz(o.in) + 4); break;
      case K_WREDUCE: bytes += (double)o.splits * params[o.w].n * 4 + params[o.w].n * 4; break;
      default: break;
    }
  }
  int run_phase(int p) { return run_phase(p, stream, 0); }
  int run_phase(int p, cudaStream_t st, int cap);
  int do_forward(bool timed);
  int do_backward(bool timed);
  int do_sgd(float lr, bool timed);
  cudaError_t refresh_wt();
  int fail(int code, const std::string& m) {
    err = m;
    return code;
  }
  int cuda_check(cudaError_t e, const char* what) {
    if (e == cudaSuccess) return PNN_OK;
    err = std::string(what) + ": " + cudaGetErrorString(e);
    return PNN_ECUDA;
  }
};

// ====================================================================== plan
int pnn_net::plan(const pnn_desc* d) {
  B = d->batch; in_c = d->in_c; in_h = d->in_h; in_w = d->in_w; classes = d->classes; N = d->n_seg;
  if (B <= 0 || B > 1024 || in_c <= 0 || in_h <= 0 || in_w <= 0 || classes <= 0 || N <= 0)
    return fail(PNN_EINVAL, "bad batch/input/classes/segments");
  int total = 0;
  for (int j = 0; j < N; ++j) {
    if (d->segments[j] <= 0) return fail(PNN_EINVAL, "empty segment");
    total += d->segments[j];
  }
  if (total != d->n_body) return fail(PNN_EINVAL, "segments do not sum to the body length");
  if (d->n_stem <= 0) return fail(PNN_EINVAL, "empty stem");
  act_dt = opt.precision == PNN_FP32_CHECK ? DT_F32 : DT_BF16;
  stream_dt = (opt.precision == PNN_FP32_CHECK || opt.stream_fp32) ? DT_F32 : DT_BF16;
  head_kind = d->head_kind;
  for (int i = 0; i < d->n_hidden; ++i) head_hidden.push_back(d->head_hidden[i]);
  auto check_layers = [&](const pnn_layer* ls, int n) -> bool {
    for (int i = 0; i < n; ++i) {
      const pnn_layer& l = ls[i];
      if (l.op < 0 || l.op > 4 || l.cout <= 0 || (l.stride != 1 && l.stride != 2)) return false;
      if ((l.op == PNN_CONV || l.op == PNN_CONV_BN_RELU) && l.k != 1 && l.k != 3) return false;
      if (l.op == PNN_BOTTLENECK && l.mid <= 0) return false;
      if (l.op == PNN_BASIC && l.stride != 1) return false;
    }
    return true;
  };
  if (!check_layers(d->stem, d->n_stem) || !check_layers(d->body, d->n_body)) return fail(PNN_EINVAL, "bad layer");

  x_in = new_value(in_c, in_h, in_w, act_dt, false);
  pre_f.resize(N); fine_f.resize(N);
  std::vector<std::vector<int>> seg_ids(N), pre_ids(N), coarse_ids(std::max(0, N - 1));
  xs.assign(N, -1); ys.assign(N, -1);
  // eq:barf order: (delta_j, phi_j) for j = 1..N, then eta_j, then eps.
  int body0 = 0;
  std::vector<std::tuple<int, int, int>> Xshape(N + 1);  // X_0..X_N (C,H,W)
  for (int j = 0; j < N; ++j) {
    PCur pc{&pre_ids[j], 0, false};
    if (j == 0) {
      xs[0] = stack(pre_f[0], d->stem, d->n_stem, x_in, pc, -100, false);
      Xshape[0] = {vals[xs[0]].C, vals[xs[0]].H, vals[xs[0]].W};
    } else {
      // C^j: 3x3/s2 maxpools down to X_{j-1}, then a 1x1 conv (+BN+ReLU)
      auto [tc, th, tw] = Xshape[j];
      int v = x_in, npool = 0;
      while (vals[v].H > th) {
        v = pool(pre_f[j], v, 3, 2, 1, -100, npool);
        ++npool;
      }
      if (vals[v].H != th || vals[v].W != tw) return fail(PNN_EINVAL, "C^j: input size is not X_{j-1} times a power of 2");
      int w = take(pc, 0, tc, in_c, 1, 1);
      int h = conv(pre_f[j], v, w, tc, 1, 1, -1, act_dt, -99, 0);
      if (d->cj_post == PNN_CJ_BN_RELU) {
        int g = take(pc, 1, tc), b = take(pc, 2, tc);
        h = bn_virtual(pre_f[j], h, g, b, true, -99, 1);
      }
      xs[j] = h;
      if (vals[h].C != tc) return fail(PNN_EINVAL, "C^j shape");
    }
    PCur ps{&seg_ids[j], 0, false};
    ys[j] = stack(fine_f[j], d->body + body0, d->segments[j], xs[j], ps, 0, true);
    body0 += d->segments[j];
    Xshape[j + 1] = {vals[ys[j]].C, vals[ys[j]].H, vals[ys[j]].W};
  }
  // coarse network, eq:correct
  const bool delta = opt.correction == PNN_CORR_DELTA;
  int cofs = 0;
  rs.assign(std::max(0, N - 1), -1);
  rts.assign(N, -1);
  y_is_r.assign(N, 0);
  rtN_in_ytilde = false;
  // The correction's sums go into the epilogue of the conv that produces
  // their first operand when that conv already adds a residual (a
  // pre-activation bottleneck or coarse RU output) and has room for more
  // addends: r_j = y_j - x_{j+1} into the last conv of g^j, rt_{j+1} = r_{j+1}
  // + F^j(rt_j) (delta form: - F^j(x_{j+1})) into the last conv of F^j,
  // ytilde = y_N + rt_N into the last conv of F^{N-1}.  (Not with the
  // coarse/fine overlap, which defers a term of the r_{N-1} backward.)
  const bool fuse = opt.fuse_correction && !(opt.overlap > 0 && opt.correction == PNN_CORR_RESIDUAL) && N > 1;
  auto free_slots = [&](int v) -> int {
    const int p = v >= 0 ? vals[v].producer : -1;
    if (!fuse || p < 0) return 0;
    const POp& o = ops[p];
    if (!((o.kind == K_CONV_FWD || o.kind == K_CONV_FWD_TC) && o.out == v && o.res >= 0)) return 0;
    return (o.res2[0] < 0) + (o.res2[1] < 0);
  };
  auto fuse_add = [&](int v, int addend, float c) {
    POp& o = ops[vals[v].producer];
    const int e = o.res2[0] < 0 ? 0 : 1;
    o.res2[e] = addend;
    o.rcoef[e] = c;
  };
  derived.clear();
  // The delta form as a chain of states s_j = x_{j+1} + rt_j: s_1 = y_1,
  // s_{j+1} = y_{j+1} + F^j(s_j) - F^j(x_{j+1}), ytilde = s_N -- the same
  // values (r_{j+1} + x_{j+2} = y_{j+1}) without r_j or a separate state sum;
  // rt_j = s_j - x_{j+1} and r_j = y_j - x_{j+1} are exported from them.
  const bool chain = fuse && delta;
  std::vector<int> f0(std::max(0, N - 1), -1);
  if (!chain) {
    for (int j = 0; j + 1 < N; ++j) {
      if (free_slots(ys[j]) >= 1) {
        fuse_add(ys[j], xs[j + 1], -1.f);
        rs[j] = ys[j];
        y_is_r[j] = 1;
        derived[{PNN_T_Y, j + 1}] = std::make_tuple(ys[j], xs[j + 1], 1.f);
      } else {
        rs[j] = ew(coarse_f, {ys[j], xs[j + 1]}, {1.f, -1.f}, false, stream_dt, 1000, j);
      }
    }
    if (N > 1) rts[0] = rs[0];
  } else {
    rts[0] = ys[0];  // s_1 = y_1
    for (int j = 0; j + 1 < N; ++j) {
      derived[{PNN_T_R, j + 1}] = std::make_tuple(ys[j], xs[j + 1], -1.f);
      derived[{PNN_T_RTILDE, j + 1}] = std::make_tuple(-1, xs[j + 1], -1.f);  // a = s_{j+1}, filled below
    }
  }
  std::vector<int> coarse_start(N, 0);
  for (int j = 0; j + 1 < N; ++j) { coarse_start[j] = cofs; cofs += d->coarse_len[j]; }
  for (int j = 0; j + 1 < N; ++j) {
    const pnn_layer* F = d->coarse + coarse_start[j];
    const int nF = d->coarse_len[j];
    if (!check_layers(F, nF) || nF <= 0) return fail(PNN_EINVAL, "bad coarse layer");
    int out;
    PCur pc{&coarse_ids[j], 0, false};
    if (!delta || chain) {
      out = stack(coarse_f, F, nF, rts[j], pc, 2000 + 100 * j, true);
      if (chain) {
        PCur pr{&coarse_ids[j], 0, true};
        delta_f.emplace_back();
        f0[j] = stack(delta_f.back(), F, nF, xs[j + 1], pr, 0, true);
      }
    } else {
      int state = ew(coarse_f, {xs[j + 1], rts[j]}, {1.f, 1.f}, false, stream_dt, 2000 + 100 * j, 99);
      out = stack(coarse_f, F, nF, state, pc, 2000 + 100 * j, true);
      // F^j(x_{j+1}) with the same parameters: independent of the chain, it
      // joins the fine wave as an extra list
      PCur pr{&coarse_ids[j], 0, true};
      delta_f.emplace_back();
      f0[j] = stack(delta_f.back(), F, nF, xs[j + 1], pr, 0, true);
    }
    if (vals[out].C != std::get<0>(Xshape[j + 2]) || vals[out].H != std::get<1>(Xshape[j + 2]))
      return fail(PNN_EINVAL, "coarse block output is not X_{j+1}");
    if (chain) {
      // s_{j+1} = y_{j+1} + F^j(s_j) - F^j(x_{j+1})
      if (free_slots(out) >= 2) {
        fuse_add(out, ys[j + 1], 1.f);
        fuse_add(out, f0[j], -1.f);
        rts[j + 1] = out;
      } else {
        rts[j + 1] = ew(coarse_f, {ys[j + 1], out, f0[j]}, {1.f, 1.f, -1.f}, false, stream_dt, 2000 + 100 * j, 98);
      }
    } else if (!delta) {
      if (j + 1 == N - 1) {
        rts[j + 1] = out;
      } else if (free_slots(out) >= 1) {
        fuse_add(out, rs[j + 1], 1.f);
        rts[j + 1] = out;
      } else {
        rts[j + 1] = ew(coarse_f, {rs[j + 1], out}, {1.f, 1.f}, false, stream_dt, 2000 + 100 * j, 98);
      }
    } else {
      if (j + 1 < N - 1) {
        if (free_slots(out) >= 2) {
          fuse_add(out, rs[j + 1], 1.f);
          fuse_add(out, f0[j], -1.f);
          rts[j + 1] = out;
        } else {
          rts[j + 1] = ew(coarse_f, {rs[j + 1], out, f0[j]}, {1.f, 1.f, -1.f}, false, stream_dt, 2000 + 100 * j, 98);
        }
      } else if (free_slots(out) >= 1) {
        fuse_add(out, f0[j], -1.f);
        rts[j + 1] = out;
      } else {
        rts[j + 1] = ew(coarse_f, {out, f0[j]}, {1.f, -1.f}, false, stream_dt, 2000 + 100 * j, 98);
      }
    }
  }
  // ytilde joins the post phase, so that its backward (which writes dL/dy_N =
  // D_N) is complete when the head's backward is
  if (chain) {
    ytilde = rts[N - 1];  // s_N
    for (int j = 0; j + 1 < N; ++j) std::get<0>(derived[{PNN_T_RTILDE, j + 1}]) = rts[j];
    derived[{PNN_T_RTILDE, N}] = std::make_tuple(ytilde, ys[N - 1], -1.f);
  } else if (N > 1 && free_slots(rts[N - 1]) >= 1) {
    fuse_add(rts[N - 1], ys[N - 1], 1.f);
    ytilde = rts[N - 1];
    rtN_in_ytilde = true;
    derived[{PNN_T_RTILDE, N}] = std::make_tuple(ytilde, ys[N - 1], -1.f);
  } else {
    ytilde = N > 1 ? ew(head_f, {ys[N - 1], rts[N - 1]}, {1.f, 1.f}, false, stream_dt, 9000, 0) : ys[0];
  }
  if (N == 1) rts[0] = ytilde;
  // head h
  std::vector<int> head_ids;
  PCur ph_{&head_ids, 0, false};
  const int Cf = vals[ytilde].C;
  head_in = ytilde;
  if (head_kind == PNN_HEAD_BN_RELU_GAP_FC) {
    int g = take(ph_, 1, Cf), b = take(ph_, 2, Cf);
    head_in = bn_virtual(head_f, ytilde, g, b, true, 9500, 0);
  } else if (head_kind != PNN_HEAD_GAP_FC && head_kind != PNN_HEAD_GAP_MLP) {
    return fail(PNN_EINVAL, "bad head kind");
  }
  if (head_kind != PNN_HEAD_GAP_MLP && !head_hidden.empty()) return fail(PNN_EINVAL, "hidden widths need gap_mlp");
  fc_width.push_back(Cf);
  for (int h : head_hidden) fc_width.push_back(h);
  fc_width.push_back(classes);
  for (size_t l = 0; l + 1 < fc_width.size(); ++l) {
    fc_w.push_back(take(ph_, 3, fc_width[l + 1], fc_width[l]));
    fc_b.push_back(take(ph_, 4, fc_width[l + 1]));
  }
  {
    POp h;
    h.kind = K_HEAD_FWD; h.in = head_in;
    h.key[0] = 9600;
    new_op(head_f, h);
  }
  // reorder the parameter table into eq:barf order
  {
    std::vector<int> order;
    for (int j = 0; j < N; ++j) {
      order.insert(order.end(), pre_ids[j].begin(), pre_ids[j].end());
      order.insert(order.end(), seg_ids[j].begin(), seg_ids[j].end());
    }
    for (int j = 0; j + 1 < N; ++j) order.insert(order.end(), coarse_ids[j].begin(), coarse_ids[j].end());
    order.insert(order.end(), head_ids.begin(), head_ids.end());
    if (order.size() != params.size()) return fail(PNN_EINVAL, "internal: parameter order");
    size_t o = 0;
    for (int id : order) { params[id].off = o; o += params[id].n; }
  }
  // the tcgen05 conv reads weight rows with 16-byte loads: a weight that does
  // not start on an 8-element boundary falls back to the CUDA-core kernel
  for (auto& c : ops) {
    if (c.kind != K_CONV_FWD_TC || params[c.w].off % 8 == 0) continue;
    c.kind = K_CONV_FWD;
    const int cout = vals[c.out].C;
    c.variant = cout <= 16 ? 2 : (cout <= 32 ? 1 : 0);
    const ConvTile t = simt_tile(c.variant);
    c.mtiles = cdiv(rows(c.out), t.BM);
    c.ntiles = cdiv(cout, t.BN);
    c.tiles = c.mtiles;
    if (c.stats_norm >= 0) {
      norms[c.stats_norm].tiles = c.tiles;
      norms[c.stats_norm].stat_rows = t.BM;
    }
  }
  // BN running statistics: one slot of 2C floats per BN layer, in the order of
  // its gamma in the parameter vector (the delta form's two evaluations of F^j
  // share their layers' slots)
  {
    std::vector<int> gam;
    for (size_t i = 0; i < params.size(); ++i)
      if (params[i].kind == 1) gam.push_back((int)i);
    std::sort(gam.begin(), gam.end(), [&](int a, int b) { return params[a].off < params[b].off; });
    run_at.assign(params.size(), 0);
    running_floats = 0;
    for (int g : gam) {
      run_at[g] = running_floats;
      running_floats += 2 * params[g].n;
    }
  }
  if (!opt.inference) {
  // backward lists (Algorithm 2): head, coarse chain, fine wave, pre wave
  overlap_on = opt.overlap > 0 && opt.correction == PNN_CORR_RESIDUAL && N > 1;
  if (overlap_on) {
    defer_x = xs[N - 1];
    defer_r = rs[N - 2];
  }
  backward_list(head_f, head_b);
  backward_list(coarse_f, coarse_b);
  delta_b.resize(delta_f.size());
  for (size_t j = 0; j < delta_f.size(); ++j) backward_list(delta_f[j], delta_b[j]);
  fine_b.resize(fine_f.size());
  if (overlap_on) {
    // the last subnetwork first (it writes dL/dx_N first), then the deferred
    // term dL/dx_N -= dL/dr_{N-1}, then the other subnetworks
    backward_list(fine_f[N - 1], fine_b[N - 1]);
    POp e;
    e.kind = K_EW_BWD;
    e.in = defer_r; e.out = defer_r; e.relu = false;
    e.nin = 1; e.ins[0] = defer_x; e.coef[0] = -1.f; e.acc_in[0] = grad_acc(defer_x);
    e.tiles = cdiv(rows(defer_x), kEwRowsPerTile);
    e.key[0] = -1000; e.key[1] = -(N - 2); e.key[2] = 1;
    new_op(fix_b, e);
    for (int j = 0; j + 1 < N; ++j) backward_list(fine_f[j], fine_b[j]);
  } else {
    for (size_t j = 0; j < fine_f.size(); ++j) backward_list(fine_f[j], fine_b[j]);
  }
  pre_b.resize(N);
  for (int j = 0; j < N; ++j) backward_list(pre_f[j], pre_b[j]);
  // gradient-accumulating parameters (delta mode: F^j used twice)
  {
    std::vector<int> seen(params.size(), 0);
    auto mark = [&](POp& o, int pid) { o.acc = seen[pid]++ ? 1 : 0; };
    auto visit = [&](std::vector<int>& L) {
      for (int id : L) {
        POp& o = ops[id];
        if (o.kind == K_WREDUCE) mark(o, o.w);
        if (o.kind == K_BNB_FIN) {
          const Norm& n = norms[o.norm];
          o.acc_in[0] = seen[n.gamma]++ ? 1 : 0;
          seen[n.beta]++;
        }
      }
    };
    visit(head_b);
    visit(coarse_b);
    for (auto& L : delta_b) visit(L);
    for (auto& L : fine_b) visit(L);
    for (auto& L : pre_b) visit(L);
  }
  }  // !opt.inference
  // ---------------------------------------------------------- memory plan
  cursor = 0;
  off_master = alloc(nparams * 4);
  off_grad = opt.inference ? 0 : alloc(nparams * 4);
  off_mom = opt.inference ? 0 : alloc(nparams * 4);
  off_shadow = act_dt == DT_BF16 ? alloc(nparams * 2) : 0;
  off_wt = act_dt == DT_BF16 ? alloc(nparams * 2) : 0;
  off_running = alloc(running_floats * 4);
  if (opt.inference) {
    share_activation_buffers();
  } else {
    for (auto& v : vals) {
      if (!v.virt) v.off = alloc((size_t)B * v.H * v.W * v.C * (v.dt == DT_F32 ? 4 : 2));
      if (v.need_grad) v.goff = alloc((size_t)B * v.H * v.W * v.C * 4);
    }
  }
  // finalize counters: one region, zeroed at bind (each launch leaves them zero)
  {
    size_t ncnt = 0;
    for (auto& n : norms) ncnt += 2 * (size_t)cdiv(n.C, 32);
    off_fin_cnt = alloc(ncnt * 4);
    fin_cnt_bytes = ncnt * 4;
    size_t at = off_fin_cnt;
    for (auto& n : norms) {
      n.fcnt = at; at += (size_t)cdiv(n.C, 32) * 4;
      n.bcnt = at; at += (size_t)cdiv(n.C, 32) * 4;
    }
  }
  for (auto& n : norms) {
    n.part = alloc((size_t)n.tiles * n.C * 8);
    n.mean = alloc(n.C * 4); n.rstd = alloc(n.C * 4); n.scale = alloc(n.C * 4); n.shift = alloc(n.C * 4);
    n.run = off_running + run_at[n.gamma] * 4;
    n.fscr = alloc((size_t)cdiv(std::max(n.tiles, 1), kFinTilesPerCta) * n.C * 16);
    if (opt.inference) continue;
    n.btiles = cdiv(n.count, bnb_rows_per_tile(n.C));
    // room for the reduce kernel's tiles or a fused data gradient's 128-row tiles
    const int bt = std::max(n.btiles, cdiv(n.count, kTcBM));
    n.bpart = alloc((size_t)bt * n.C * 8);
    n.bscr = alloc((size_t)cdiv(bt, kFinTilesPerCta) * n.C * 16);
    n.coef = alloc((size_t)n.C * 12);
  }
  // wgrad scratch: one region per op (sized per op)
  for (auto& o : ops)
    if (o.kind == K_WGRAD || o.kind == K_WGRAD_TC) o.scratch = alloc((size_t)o.splits * vals[o.out].C * o.k * o.k * vals[o.in].C * 4);
  for (size_t l = 0; l < fc_width.size(); ++l) {
    feat.push_back(alloc((size_t)B * fc_width[l] * 4));
    dfeat.push_back(alloc((size_t)B * fc_width[l] * 4));
  }
  loss_off = alloc(64);
  status_off = alloc(64);
  labels_stage = alloc((size_t)B * 4);
  x_stage = alloc((size_t)B * in_c * in_h * in_w * 4);
  size_t biggest = (size_t)B * classes;
  for (auto& v : vals) biggest = std::max(biggest, (size_t)B * v.H * v.W * v.C);
  export_off = alloc(biggest * 4);
  export_bytes = biggest * 4;
  return PNN_OK;
}

// ====================================================================== tables

static Src make_src(const pnn_net& n, int v) {
  Src s{};
  const Value& val = n.vals[v];
  if (val.virt) {
    const Value& h = n.vals[val.src];
    const Norm& nm = n.norms[val.norm];
    s.ptr = n.ws + h.off; s.dt = h.dt;
    s.scale = n.P<float>(nm.scale); s.shift = n.P<float>(nm.shift);
    s.relu = val.relu;
  } else {
    s.ptr = n.ws + val.off; s.dt = val.dt;
    s.scale = nullptr; s.shift = nullptr; s.relu = 0;
  }
  return s;
}

std::vector<Group> pnn_net::phase_groups(int p) const {
  // merge per-subnetwork lists by key into launch groups
  auto keyless = [&](int a, int b) {
    const POp &x = ops[a], &y = ops[b];
    return std::lexicographical_compare(x.key, x.key + 3, y.key, y.key + 3);
  };
  auto merge = [&](const std::vector<std::vector<int>>& lists) {
    std::vector<Group> groups;
    std::vector<size_t> pos(lists.size(), 0);
    while (true) {
      int best = -1;
      for (size_t i = 0; i < lists.size(); ++i)
        if (pos[i] < lists[i].size() && (best < 0 || keyless(lists[i][pos[i]], lists[best][pos[best]]))) best = (int)i;
      if (best < 0) break;
      const POp& b = ops[lists[best][pos[best]]];
      std::vector<Group> step;
      for (size_t i = 0; i < lists.size(); ++i) {
        if (pos[i] >= lists[i].size()) continue;
        const POp& o = ops[lists[i][pos[i]]];
        if (std::equal(o.key, o.key + 3, b.key)) {
          bool placed = false;
          for (auto& g : step)
            if (g.kind == o.kind && g.variant == o.variant) { g.ops.push_back(lists[i][pos[i]]); placed = true; break; }
          if (!placed) step.push_back(Group{o.kind, o.variant, {lists[i][pos[i]]}});
          pos[i]++;
        }
      }
      for (auto& g : step) groups.push_back(g);
    }
    return groups;
  };
  auto single = [&](const std::vector<int>& L) {
    std::vector<Group> g;
    for (int id : L) g.push_back(Group{ops[id].kind, ops[id].variant, {id}});
    return g;
  };
  switch (p) {
    case 0: return merge(pre_f);
    case 1: {
      std::vector<std::vector<int>> fwd_lists = fine_f;
      fwd_lists.insert(fwd_lists.end(), delta_f.begin(), delta_f.end());
      return merge(fwd_lists);
    }
    case 2: return single(coarse_f);
    case 3: return single(head_f);
    case 4: return single(head_b);
    case 5: return single(coarse_b);
    case 6: return merge(delta_b);
    case 7:
      if (overlap_on) return merge(std::vector<std::vector<int>>(fine_b.begin(), fine_b.end() - 1));
      return merge(fine_b);
    case 8: return merge(pre_b);
    case 9:
      if (overlap_on) return merge(std::vector<std::vector<int>>(fine_b.end() - 1, fine_b.end()));
      return {};
    default: return single(fix_b);
  }
}

int pnn_net::build_tables() {
  std::vector<Group> phases[11];
  for (int p = 0; p < 11; ++p) phases[p] = phase_groups(p);
  host_tables.clear();
  auto put = [&](const void* p, size_t n) { return put_table(p, n); };
  float* master = P<float>(off_master);
  float* grad = P<float>(off_grad);
  const void* wts = act_dt == DT_BF16 ? (const void*)(ws + off_shadow) : (const void*)master;
  const int wdt = act_dt;
  auto wptr = [&](int pid) -> const void* {
    return (const char*)wts + params[pid].off * (wdt == DT_BF16 ? 2 : 4);
  };
  for (int p = 0; p < 11; ++p) {
    ph[p].launches.clear();
    for (auto& g : phases[p]) {
      std::vector<uint8_t> tab;
      std::vector<int> tstart;
      int total = 0;
      auto add = [&](const void* d, size_t sz, int tiles) {
        size_t o = tab.size();
        tab.resize(o + sz);
        memcpy(tab.data() + o, d, sz);
        tstart.push_back(total);
        total += tiles;
      };
      for (int id : g.ops) {
        const POp& o = ops[id];
        switch (o.kind) {
          case K_CONV_FWD:
          case K_CONV_FWD_TC:
          case K_DGRAD:
          case K_DGRAD_TC:
          case K_WGRAD:
          case K_WGRAD_TC: {
            ConvDesc c{};
            const Value& iv = vals[o.in];
            const Value& ov = vals[o.out];
            c.x = make_src(*this, o.in);
            c.w = wptr(o.w); c.w_dt = wdt;
            c.B = B; c.H = iv.H; c.W = iv.W; c.C = iv.C; c.P = ov.H; c.Q = ov.W; c.K = ov.C;
            c.R = o.k; c.S = o.k; c.stride = o.stride; c.pad = o.pad;
            c.mtiles = o.mtiles; c.ntiles = o.ntiles;
            c.ntile_w = tc_ntile_w(o.kind, o.variant);
            c.mtile_rows = tc_mtile_rows(o.kind, o.variant, iv.C);
            c.op_bf16 = act_dt == DT_BF16 && ((o.kind != K_DGRAD && o.kind != K_WGRAD) || !opt.grad_fp32);
            if (o.kind == K_DGRAD_TC) c.w = (const char*)(ws + off_wt) + params[o.w].off * 2;
            if ((o.kind == K_CONV_FWD_TC || o.kind == K_DGRAD_TC) && o.variant == 1) {
              const bool fwd = o.kind == K_CONV_FWD_TC;
              const int ch = fwd ? iv.C : ov.C;            // channels of the A source
              const int ncols = fwd ? ov.C : iv.C;          // GEMM N
              const int kt = o.k * o.k * ch;
              const void* a_src = fwd ? c.x.ptr : (const void*)P<float>(gptr(o.out));
              const bool a_bf16 = fwd && c.x.dt == DT_BF16;
              const int64_t a_rows = fwd ? (int64_t)B * iv.H * iv.W : (int64_t)B * ov.H * ov.W;
              const int bn = o.ntiles == 1 ? ((ncols + 15) & ~15) : tc_ntile_w(o.kind, o.variant);
              // a third map over the output for the epilogue's TMA stores, a
              // fourth (halo tiles) over the A source with one box per tile
              const int aW = fwd ? iv.W : ov.W, aH = fwd ? iv.H : ov.H;
              const bool halo = use_halo(opt.conv_impl, fwd ? 0 : 1, o.k, o.stride, o.pad, aH, aW, ch, bn);
              CUtensorMap maps[4];
              memset(maps, 0, sizeof maps);
              if (ws) {
                int r = encode_map(&maps[0], a_src, a_bf16, ch, a_rows, std::min(ch, 64), kTcBM, 0);
                if (!r) r = encode_map(&maps[1], c.w, true, kt, ncols, 64, bn, 128);
                if (!r && fwd)
                  r = encode_map(&maps[2], ws + ov.off, ov.dt == DT_BF16, ov.C, (int64_t)B * ov.H * ov.W, 16, 32,
                                 ov.dt == DT_BF16 ? 32 : 64);
                if (!r && !fwd)  // data gradient: dx [pixels][C] fp32, stored or reduce-added
                  r = encode_map(&maps[2], P<float>(gptr(o.in)), false, iv.C, (int64_t)B * iv.H * iv.W, 16, 32, 64);
                if (!r && halo) r = encode_map(&maps[3], a_src, a_bf16, ch, a_rows, ch, halo_rows(aW), 0);
                if (r) return r;
              }
              const size_t mo = put(maps, sizeof maps);
              c.tma_a = ws ? ws + tables_off + mo : nullptr;
              c.tma_b = ws ? ws + tables_off + mo + sizeof(CUtensorMap) : nullptr;
              c.tma_y = ws ? ws + tables_off + mo + 2 * sizeof(CUtensorMap) : nullptr;
              c.tma_h = ws && halo ? ws + tables_off + mo + 3 * sizeof(CUtensorMap) : nullptr;
            }
            if (o.kind == K_WGRAD_TC && o.variant == 1) {
              // activation halo box [hrows][cwx] (its dtype), gradient box [64][K] fp32
              const WgBoxes bx = wg_boxes(iv.C, ov.C, iv.W, o.pad, c.x.dt == DT_BF16);
              CUtensorMap maps[2];
              memset(maps, 0, sizeof maps);
              if (ws) {
                int r = encode_map(&maps[0], c.x.ptr, c.x.dt == DT_BF16, iv.C, (int64_t)B * iv.H * iv.W, bx.cwx,
                                   bx.hrows, 0);
                if (!r) r = encode_map(&maps[1], P<float>(gptr(o.out)), false, ov.C, (int64_t)B * ov.H * ov.W, ov.C,
                                       64, 0);
                if (r) return r;
              }
              const size_t mo = put(maps, sizeof maps);
              c.tma_a = ws ? ws + tables_off + mo : nullptr;
              c.tma_b = ws ? ws + tables_off + mo + sizeof(CUtensorMap) : nullptr;
            }
            if (o.kind == K_CONV_FWD || o.kind == K_CONV_FWD_TC) {
              c.y = ws + ov.off; c.y_dt = ov.dt;
              if (o.res >= 0) { c.res = ws + vals[o.res].off; c.res_dt = vals[o.res].dt; }
              for (int e = 0; e < 2; ++e)
                if (o.res2[e] >= 0) {
                  c.res2[e] = ws + vals[o.res2[e]].off;
                  c.res2_dt[e] = vals[o.res2[e]].dt;
                  c.res2_c[e] = o.rcoef[e];
                }
              if (o.stats_norm >= 0) c.stats = P<float>(norms[o.stats_norm].part);
              add(&c, sizeof c, o.mtiles * o.ntiles);
            } else if (o.kind == K_DGRAD || o.kind == K_DGRAD_TC) {
              c.dy = P<float>(gptr(o.out));
              c.dx = P<float>(gptr(o.in)); c.accumulate = o.acc;
              if (o.bn_fuse >= 0) {
                const Norm& nf = norms[o.bn_fuse];
                c.bn_mean = P<float>(nf.mean); c.bn_rstd = P<float>(nf.rstd); c.bnb_part = P<float>(nf.bpart);
              }
              add(&c, sizeof c, o.tiles);
            } else {
              c.dy = P<float>(gptr(o.out));
              c.dw_part = P<float>(o.scratch);
              c.splits = o.splits; c.pix_per_split = o.pix_per_split;
              add(&c, sizeof c, o.tiles);
            }
            break;
          }
          case K_WREDUCE: {
            // find the matching wgrad scratch: the op right before in the same list
            WReduceDesc r{};
            const POp* wg = nullptr;
            for (int q = id - 1; q >= 0; --q)
              if ((ops[q].kind == K_WGRAD || ops[q].kind == K_WGRAD_TC) && ops[q].w == o.w && ops[q].out == o.out) {
                wg = &ops[q];
                break;
              }
            r.part = P<float>(wg->scratch);
            r.dw = grad + params[o.w].off;
            r.splits = o.splits;
            r.accumulate = o.acc;
            r.transposed = wg->kind == K_WGRAD_TC;
            r.kout = vals[o.out].C;
            r.rsc = o.k * o.k * vals[o.in].C;
            r.n = (int64_t)params[o.w].n;
            r.tiles = o.tiles;
            add(&r, sizeof r, o.tiles);
            break;
          }
          case K_EW: {
            EwDesc e{};
            for (int i = 0; i < o.nin; ++i) { e.in[i] = make_src(*this, o.ins[i]); e.coef[i] = o.coef[i]; }
            e.nin = o.nin;
            const int ref = o.out >= 0 ? o.out : o.ins[0];
            if (o.out >= 0) { e.out = ws + vals[o.out].off; e.out_dt = vals[o.out].dt; }
            e.relu = o.relu;
            if (o.stats_norm >= 0) e.stats = P<float>(norms[o.stats_norm].part);
            e.M = rows(ref); e.C = vals[ref].C;
            e.rows_per_tile = kEwRowsPerTile; e.tiles = o.tiles;
            add(&e, sizeof e, o.tiles);
            break;
          }
          case K_EW_BWD: {
            EwBwdDesc e{};
            e.dout = P<float>(gptr(o.in));
            if (o.out >= 0) { e.out = ws + vals[o.out].off; e.out_dt = vals[o.out].dt; }
            e.relu = o.relu;
            for (int i = 0; i < o.nin; ++i) {
              e.gin[i] = P<float>(gptr(o.ins[i]));
              e.coef[i] = o.coef[i];
              e.acc[i] = o.acc_in[i];
            }
            e.nin = o.nin;
            e.M = rows(o.in); e.C = vals[o.in].C;
            e.rows_per_tile = kEwRowsPerTile; e.tiles = o.tiles;
            add(&e, sizeof e, o.tiles);
            break;
          }
          case K_BN_FIN: {
            const Norm& n = norms[o.norm];
            BnFinDesc f{};
            f.part = P<float>(n.part); f.tiles = n.tiles; f.C = n.C; f.count = n.count;
            f.rows_per_tile = n.stat_rows;
            f.gamma = master + params[n.gamma].off; f.beta = master + params[n.beta].off;
            f.mean = P<float>(n.mean); f.rstd = P<float>(n.rstd); f.scale = P<float>(n.scale); f.shift = P<float>(n.shift);
            f.run_mean = P<float>(n.run); f.run_var = P<float>(n.run) + n.C;
            f.momentum = opt.bn_momentum;
            f.eval = opt.inference ? 1 : 0;
            f.scratch = P<double>(n.fscr); f.counter = P<int32_t>(n.fcnt);
            f.cgroups = cdiv(n.C, 32);
            f.nchunk = f.eval ? 1 : cdiv(std::max(n.tiles, 1), kFinTilesPerCta);
            add(&f, sizeof f, f.cgroups * f.nchunk);
            break;
          }
          case K_BNB_RED:
          case K_BNB_FIN:
          case K_BNB_APPLY: {
            const Norm& n = norms[o.norm];
            const Value& hv = vals[n.h];
            BnBwdDesc b{};
            b.da = P<float>(gptr(o.in));
            b.h = ws + hv.off; b.h_dt = hv.dt;
            b.mean = P<float>(n.mean); b.rstd = P<float>(n.rstd); b.scale = P<float>(n.scale); b.shift = P<float>(n.shift);
            b.gamma = master + params[n.gamma].off;
            b.relu = vals[o.in].relu;
            b.part = P<float>(n.bpart);
            b.dgamma = grad + params[n.gamma].off; b.dbeta = grad + params[n.beta].off;
            b.coef = P<float>(n.coef);
            b.M = n.count; b.C = n.C;
            b.rows_per_tile = bnb_rows_per_tile(n.C); b.tiles = n.fused_tiles ? n.fused_tiles : n.btiles;
            b.scratch = P<double>(n.bscr); b.counter = P<int32_t>(n.bcnt);
            b.cgroups = cdiv(n.C, 32);
            b.nchunk = cdiv(std::max(b.tiles, 1), kFinTilesPerCta);
            if (o.kind == K_BNB_FIN) b.accumulate = o.acc_in[0];
            if (o.kind == K_BNB_APPLY) {
              b.dh = P<float>(gptr(n.h));
              b.accumulate = o.acc;
              b.add0 = o.addv[0] >= 0 ? P<float>(gptr(o.addv[0])) : nullptr;
              b.add1 = o.addv[1] >= 0 ? P<float>(gptr(o.addv[1])) : nullptr;
              b.add_c[0] = o.addc[0];
              b.add_c[1] = o.addc[1];
            }
            add(&b, sizeof b, o.kind == K_BNB_FIN ? b.cgroups * b.nchunk : o.tiles);
            break;
          }
          case K_POOL_FWD:
          case K_POOL_BWD: {
            PoolDesc q{};
            const Value& iv = vals[o.in];
            const Value& ov = vals[o.out];
            q.x = make_src(*this, o.in);
            q.y = ws + ov.off; q.y_dt = ov.dt;
            q.B = B; q.H = iv.H; q.W = iv.W; q.C = iv.C; q.P = ov.H; q.Q = ov.W; q.k = o.k; q.stride = o.stride; q.pad = o.pad;
            if (o.kind == K_POOL_BWD) {
              q.dy = P<float>(gptr(o.out)); q.dx = P<float>(gptr(o.in)); q.accumulate = o.acc;
            }
            q.tiles = o.tiles;
            add(&q, sizeof q, o.tiles);
            break;
          }
          case K_HEAD_FWD:
          case K_HEAD_BWD: {
            int v = o.in;
            add(&v, sizeof v, 1);
            break;
          }
        }
      }
      Launch L;
      L.kind = g.kind; L.variant = g.variant; L.count = (int)g.ops.size(); L.total = total; L.phase = p;
      L.flops = 0; L.bytes = 0; L.aux = 16;
      {
        const POp& o = ops[g.ops[0]];
        if (p == 1) L.block = o.key[0];
        if (p == 7) L.block = -o.key[0];
        const bool conv = o.kind == K_CONV_FWD || o.kind == K_CONV_FWD_TC || o.kind == K_DGRAD ||
                          o.kind == K_DGRAD_TC || o.kind == K_WGRAD || o.kind == K_WGRAD_TC;
        const int v = o.in >= 0 ? o.in : (o.out >= 0 ? o.out : o.ins[0]);
        for (int& x : L.shape) x = 0;
        if (conv) {
          const int sh[6] = {vals[o.in].C, vals[o.out].C, o.k, o.stride, vals[o.out].H, vals[o.out].W};
          for (int i = 0; i < 6; ++i) L.shape[i] = sh[i];
        } else if (v >= 0 && v < (int)vals.size()) {
          L.shape[0] = vals[v].C; L.shape[1] = vals[v].H; L.shape[2] = vals[v].W;
        }
      }
      L.esz = 2;
      for (int id : g.ops)
        if (ops[id].kind == K_CONV_FWD_TC || ops[id].kind == K_DGRAD_TC || ops[id].kind == K_WGRAD_TC) {
          const int K = ops[id].kind == K_DGRAD_TC ? vals[ops[id].in].C : vals[ops[id].out].C;
          L.aux = std::max(L.aux, ops[id].ntiles == 1 ? ((K + 15) & ~15) : tc_ntile_w(ops[id].kind, ops[id].variant));
          if (ops[id].kind == K_DGRAD_TC) L.esz = 4;
          else if (ops[id].kind == K_CONV_FWD_TC) {
            const int src = vals[ops[id].in].virt ? vals[ops[id].in].src : ops[id].in;
            if (vals[src].dt == DT_F32) L.esz = 4;
          } else if (ops[id].variant == 1) {
            const int src = vals[ops[id].in].virt ? vals[ops[id].in].src : ops[id].in;
            const WgBoxes b = wg_boxes(vals[ops[id].in].C, vals[ops[id].out].C, vals[ops[id].in].W, ops[id].pad,
                                       vals[src].dt == DT_BF16);
            L.raw = std::max(L.raw, wg_raw_bytes(b));
          }
        }
      if (g.kind == K_CONV_FWD_TC || g.kind == K_DGRAD_TC) {
        // per instance: one tap box per k-step, or (halo tiles) one halo box per tile
        L.raw = 1024;
        for (int id : g.ops) {
          const POp& o = ops[id];
          const bool fwd = o.kind == K_CONV_FWD_TC;
          const Value& av = fwd ? vals[o.in] : vals[o.out];  // the A source
          const int ncols = fwd ? vals[o.out].C : vals[o.in].C;
          const int bn = o.ntiles == 1 ? ((ncols + 15) & ~15) : tc_ntile_w(o.kind, o.variant);
          if (g.variant == 1 && use_halo(opt.conv_impl, fwd ? 0 : 1, o.k, o.stride, o.pad, av.H, av.W, av.C, bn)) {
            L.raw = std::max(L.raw, halo_raw_bytes(av.W, av.C, L.esz));
            L.op = std::max(L.op, halo_op_bytes(av.W, av.C, bn));
          } else {
            L.raw = std::max(L.raw, kTcBM * 64 * L.esz);
          }
        }
        if (L.op > 0) L.op = std::max(L.op, conv_tma_op_bytes(conv_mode(g.kind), L.aux));
      }
      if ((g.kind == K_CONV_FWD_TC || g.kind == K_DGRAD_TC) && g.variant == 1) {
        L.wide = 1;
        for (int id : g.ops) {
          const POp& o = ops[id];
          const int ch = o.kind == K_CONV_FWD_TC ? vals[o.in].C : vals[o.out].C;  // channels of the A source
          if (o.k * o.k * ch > 64) L.wide = 0;
        }
      }
      for (int id : g.ops) op_cost(ops[id], L.flops, L.bytes);
      tstart.push_back(total);
      L.table_off = put(tab.data(), tab.size());
      L.tstart_off = put(tstart.data(), tstart.size() * sizeof(int));
      // head ops keep their op id in the table (host-side interpretation)
      if (g.kind == K_HEAD_FWD || g.kind == K_HEAD_BWD) L.variant = g.ops[0];
      ph[p].launches.push_back(L);
    }
  }
  build_head_tables();
  {
    std::vector<WtDesc> wt;
    std::vector<int> ts;
    wt_total = 0;
    if (act_dt == DT_BF16)
      for (const ParamT& p : params) {
        if (p.kind != 0) continue;
        WtDesc w{};
        w.src = ws + off_shadow + p.off * 2;
        w.dst = ws + off_wt + p.off * 2;
        w.K = p.dims[0]; w.C = p.dims[1]; w.RS = p.dims[2] * p.dims[3];
        w.n = (int64_t)p.n;
        wt.push_back(w);
        ts.push_back(wt_total);
        wt_total += cdiv(w.n, 256);
      }
    ts.push_back(wt_total);
    wt_count = (int)wt.size();
    wt_tab = put_table(wt.data(), wt.size() * sizeof(WtDesc));
    wt_ts = put_table(ts.data(), ts.size() * sizeof(int));
  }
  counts[0] = counts[1] = 0;
  for (int p = 0; p < 4; ++p) counts[0] += (int)ph[p].launches.size();
  for (int p = 4; p < 11; ++p) counts[1] += (int)ph[p].launches.size();
  counts[2] = act_dt == DT_BF16 && wt_count ? 2 : 1;
  return PNN_OK;
}

// ====================================================================== head
void pnn_net::build_head_tables() {
  const int nfc = (int)fc_width.size() - 1;
  float* master = P<float>(off_master);
  float* grad = P<float>(off_grad);
  head_fwd_tab.clear(); head_dw_tab.clear(); head_din_tab.clear();
  int ts[2];
  for (int l = 0; l < nfc; ++l) {
    const int wi = fc_width[l], wo = fc_width[l + 1];
    GemmDesc f{};  // feat[l+1][b][o] = sum_i feat[l][b][i] W[o][i] + bias[o]
    f.A = P<float>(feat[l]); f.sam = wi; f.sak = 1;
    f.Bm = master + params[fc_w[l]].off; f.sbk = 1; f.sbn = wi;
    f.Cm = P<float>(feat[l + 1]); f.scm = wo;
    f.bias = master + params[fc_b[l]].off;
    f.M = B; f.N = wo; f.K = wi; f.relu = l + 1 < nfc;
    f.mtiles = cdiv(B, 64); f.ntiles = cdiv(wo, 64);
    head_fwd_tab.push_back(put_table(&f, sizeof f));
    GemmDesc g{};  // dW[o][i] = sum_b dfeat[l+1][b][o] feat[l][b][i]
    g.A = P<float>(dfeat[l + 1]); g.sam = 1; g.sak = wo;
    g.Bm = P<float>(feat[l]); g.sbk = wi; g.sbn = 1;
    g.Cm = grad + params[fc_w[l]].off; g.scm = wi;
    g.M = wo; g.N = wi; g.K = B;
    g.mtiles = cdiv(wo, 64); g.ntiles = cdiv(wi, 64);
    head_dw_tab.push_back(put_table(&g, sizeof g));
    GemmDesc h{};  // dfeat[l][b][i] = sum_o dfeat[l+1][b][o] W[o][i]
    h.A = P<float>(dfeat[l + 1]); h.sam = wo; h.sak = 1;
    h.Bm = master + params[fc_w[l]].off; h.sbk = wi; h.sbn = 1;
    h.Cm = P<float>(dfeat[l]); h.scm = wi;
    h.M = B; h.N = wi; h.K = wo;
    h.mtiles = cdiv(B, 64); h.ntiles = cdiv(wi, 64);
    head_din_tab.push_back(put_table(&h, sizeof h));
  }
  ts[0] = 0; ts[1] = 1 << 30;
  head_tstart = put_table(ts, sizeof ts);
}

int pnn_net::run_head_fwd() {
  const int nfc = (int)fc_width.size() - 1;
  const Value& hv = vals[head_in];
  const char* tb = ws + tables_off;
  const int* tst = reinterpret_cast<const int*>(tb + head_tstart);
  cudaError_t e = launch_gap(make_src(*this, head_in), P<float>(feat[0]), B, hv.H * hv.W, hv.C, stream);
  for (int l = 0; l < nfc && e == cudaSuccess; ++l) {
    const int wo = fc_width[l + 1];
    e = launch_gemm(reinterpret_cast<const GemmDesc*>(tb + head_fwd_tab[l]), tst, 1, cdiv(B, 64) * cdiv(wo, 64), stream);
  }
  if (e == cudaSuccess && !opt.inference)
    e = launch_softmax_ce(P<float>(feat[nfc]), labels_dev, B, classes, P<float>(loss_off), P<float>(dfeat[nfc]),
                          P<int32_t>(status_off), stream);
  return cuda_check(e, "head forward");
}

int pnn_net::run_head_bwd(int opid) {
  const int nfc = (int)fc_width.size() - 1;
  const char* tb = ws + tables_off;
  const int* tst = reinterpret_cast<const int*>(tb + head_tstart);
  float* grad = P<float>(off_grad);
  cudaError_t e = cudaSuccess;
  for (int l = nfc - 1; l >= 0 && e == cudaSuccess; --l) {
    const int wi = fc_width[l], wo = fc_width[l + 1];
    e = launch_gemm(reinterpret_cast<const GemmDesc*>(tb + head_dw_tab[l]), tst, 1, cdiv(wo, 64) * cdiv(wi, 64), stream);
    if (e == cudaSuccess) e = launch_colsum(P<float>(dfeat[l + 1]), B, wo, grad + params[fc_b[l]].off, stream);
    if (e == cudaSuccess)
      e = launch_gemm(reinterpret_cast<const GemmDesc*>(tb + head_din_tab[l]), tst, 1, cdiv(B, 64) * cdiv(wi, 64), stream);
    if (e == cudaSuccess && l > 0) e = launch_relu_mask(P<float>(dfeat[l]), P<float>(feat[l]), (int64_t)B * wi, stream);
  }
  const Value& hv = vals[head_in];
  (void)opid;
  if (e == cudaSuccess) e = launch_gap_bwd(P<float>(dfeat[0]), P<float>(gptr(head_in)), B, hv.H * hv.W, hv.C, stream);
  return cuda_check(e, "head backward");
}

// ====================================================================== execution
int pnn_net::run_phase(int p, cudaStream_t st, int cap) {
  const char* tb = ws + tables_off;
  for (const Launch& L : ph[p].launches) {
    const void* tab = tb + L.table_off;
    const int* ts = reinterpret_cast<const int*>(tb + L.tstart_off);
    cudaError_t e = cudaSuccess;
    if (prof) {
      if (pnext + 2 > pev.size()) {
        size_t old = pev.size();
        pev.resize(std::max<size_t>(2 * old, 4096));
        for (size_t i = old; i < pev.size(); ++i) cudaEventCreate(&pev[i]);
        plaunch.resize(pev.size() / 2);
      }
      plaunch[pnext / 2] = &L;
      cudaEventRecord(pev[pnext], st);
    }
    switch (L.kind) {
      case K_CONV_FWD: e = launch_conv_fwd_simt((const ConvDesc*)tab, ts, L.count, L.total, L.variant, st); break;
      case K_CONV_FWD_TC:
        e = L.variant == 1
                ? launch_conv_tma(0, L.wide, (const ConvDesc*)tab, ts, L.count, L.total, L.aux, L.raw, L.op,
                                  P<int32_t>(status_off), st, cap)
                : launch_conv_fwd_tc((const ConvDesc*)tab, ts, L.count, L.total, L.aux, P<int32_t>(status_off), st, cap);
        break;
      case K_DGRAD_TC:
        e = L.variant == 1
                ? launch_conv_tma(1, L.wide, (const ConvDesc*)tab, ts, L.count, L.total, L.aux, L.raw, L.op,
                                  P<int32_t>(status_off), st, cap)
                : launch_conv_dgrad_tc((const ConvDesc*)tab, ts, L.count, L.total, L.aux, P<int32_t>(status_off),
                                       st, cap);
        break;
      case K_WGRAD_TC:
        e = L.variant == 1
                ? launch_conv_tma(2, L.wide, (const ConvDesc*)tab, ts, L.count, L.total, L.aux, L.raw, L.op,
                                  P<int32_t>(status_off), st, cap)
                : launch_conv_wgrad_tc((const ConvDesc*)tab, ts, L.count, L.total, L.aux, P<int32_t>(status_off),
                                       st, cap);
        break;
      case K_DGRAD: e = launch_conv_dgrad_simt((const ConvDesc*)tab, ts, L.count, L.total, L.variant, st); break;
      case K_WGRAD: e = launch_conv_wgrad_simt((const ConvDesc*)tab, ts, L.count, L.total, L.variant, st); break;
      case K_WREDUCE: e = launch_wreduce((const WReduceDesc*)tab, ts, L.count, L.total, st); break;
      case K_EW: e = launch_ew((const EwDesc*)tab, ts, L.count, L.total, st); break;
      case K_EW_BWD: e = launch_ew_bwd((const EwBwdDesc*)tab, ts, L.count, L.total, st); break;
      case K_BN_FIN: e = launch_bn_fin((const BnFinDesc*)tab, ts, L.count, L.total, st); break;
      case K_BNB_RED:
        e = L.variant ? launch_bnb_reduce8((const BnBwdDesc*)tab, ts, L.count, L.total, st)
                      : launch_bnb_reduce((const BnBwdDesc*)tab, ts, L.count, L.total, st);
        break;
      case K_BNB_FIN: e = launch_bnb_fin((const BnBwdDesc*)tab, ts, L.count, L.total, st); break;
      case K_BNB_APPLY:
        e = L.variant ? launch_bnb_apply8((const BnBwdDesc*)tab, ts, L.count, L.total, st)
                      : launch_bnb_apply((const BnBwdDesc*)tab, ts, L.count, L.total, st);
        break;
      case K_POOL_FWD: e = launch_pool_fwd((const PoolDesc*)tab, ts, L.count, L.total, st); break;
      case K_POOL_BWD: e = launch_pool_bwd((const PoolDesc*)tab, ts, L.count, L.total, st); break;
      case K_HEAD_FWD: { int r = run_head_fwd(); if (r) return r; break; }
      case K_HEAD_BWD: { int r = run_head_bwd(L.variant); if (r) return r; break; }
      default: return fail(PNN_EINVAL, "internal: unknown launch kind");
    }
    if (e != cudaSuccess) return cuda_check(e, "kernel launch");
    if (prof) {
      cudaEventRecord(pev[pnext + 1], st);
      pnext += 2;
    }
  }
  return PNN_OK;
}

int pnn_net::do_forward(bool timed) {
  if (timed) cudaEventRecord(ev[0], stream);
  cudaError_t e = launch_pack_input(x_dev, ws + vals[x_in].off, vals[x_in].dt, B, in_c, in_h, in_w, stream);
  if (e != cudaSuccess) return cuda_check(e, "pack input");
  for (int p = 0; p < 4; ++p) {
    int r = run_phase(p);
    if (r) return r;
    if (timed) cudaEventRecord(ev[p + 1], stream);
  }
  return PNN_OK;
}

int pnn_net::do_backward(bool timed) {
  if (timed) cudaEventRecord(ev[5], stream);
  if (overlap_on) {
    int r = run_phase(4);
    if (r) return r;
    if (timed) cudaEventRecord(ev[6], stream);
    // fork: the coarse chain on the high-priority stream, the last subnetwork's
    // backward (it needs only D_N) beside it with a capped grid; then join
    cudaError_t e = cudaEventRecord(fork_ev, stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s_hi, fork_ev, 0);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s_lo, fork_ev, 0);
    if (e != cudaSuccess) return cuda_check(e, "fork");
    r = run_phase(9, s_lo, lo_cap);
    if (!r) r = run_phase(5, s_hi, 0);
    if (r) return r;
    e = cudaEventRecord(hi_done, s_hi);
    if (e == cudaSuccess) e = cudaEventRecord(lo_done, s_lo);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(stream, hi_done, 0);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(stream, lo_done, 0);
    if (e != cudaSuccess) return cuda_check(e, "join");
    if (timed) cudaEventRecord(ev[7], stream);
    for (int p : {6, 10, 7}) {
      r = run_phase(p);
      if (r) return r;
    }
    if (timed) cudaEventRecord(ev[8], stream);
    r = run_phase(8);
    if (r) return r;
    if (timed) cudaEventRecord(ev[9], stream);
    return PNN_OK;
  }
  for (int p = 4; p < 9; ++p) {
    int r = run_phase(p);
    if (r) return r;
    // phase -> event: head 6, coarse 7, (delta+fine) 8, pre 9
    if (timed && p != 6) cudaEventRecord(ev[p == 4 ? 6 : (p == 5 ? 7 : (p == 7 ? 8 : 9))], stream);
  }
  return PNN_OK;
}

cudaError_t pnn_net::refresh_wt() {
  if (act_dt != DT_BF16 || wt_count == 0) return cudaSuccess;
  const char* tb = ws + tables_off;
  return launch_wtrans(reinterpret_cast<const WtDesc*>(tb + wt_tab), reinterpret_cast<const int*>(tb + wt_ts), wt_count,
                       wt_total, stream);
}

int pnn_net::do_sgd(float lr, bool timed) {
  if (timed) cudaEventRecord(ev[10], stream);
  if (lr <= 0.f) lr = opt.lr;
  cudaError_t e = launch_sgd(P<float>(off_master), P<float>(off_grad), P<float>(off_mom),
                             act_dt == DT_BF16 ? (void*)(ws + off_shadow) : nullptr, DT_BF16, (int64_t)nparams, lr,
                             opt.momentum, opt.weight_decay, opt.nesterov, first_step ? 1 : 0, stream);
  if (e == cudaSuccess) e = refresh_wt();
  if (timed) cudaEventRecord(ev[11], stream);
  first_step = false;
  return cuda_check(e, "sgd");
}

// ---------------------------------------------------------------- host helpers
namespace {
// theta-bar (K,C,R,S) <-> internal (K,R,S,C) for conv weights
void to_internal(const ParamT& p, const float* src, float* dst) {
  if (p.kind != 0 || (p.dims[2] == 1 && p.dims[3] == 1)) {
    memcpy(dst, src, p.n * 4);
    return;
  }
  const int K = p.dims[0], C = p.dims[1], R = p.dims[2], S = p.dims[3];
  for (int k = 0; k < K; ++k)
    for (int c = 0; c < C; ++c)
      for (int r = 0; r < R; ++r)
        for (int s = 0; s < S; ++s) dst[((k * R + r) * S + s) * C + c] = src[((k * C + c) * R + r) * S + s];
}
void to_external(const ParamT& p, const float* src, float* dst) {
  if (p.kind != 0 || (p.dims[2] == 1 && p.dims[3] == 1)) {
    memcpy(dst, src, p.n * 4);
    return;
  }
  const int K = p.dims[0], C = p.dims[1], R = p.dims[2], S = p.dims[3];
  for (int k = 0; k < K; ++k)
    for (int c = 0; c < C; ++c)
      for (int r = 0; r < R; ++r)
        for (int s = 0; s < S; ++s) dst[((k * C + c) * R + r) * S + s] = src[((k * R + r) * S + s) * C + c];
}
uint64_t splitmix64(uint64_t& s) {
  uint64_t z = (s += 0x9E3779B97F4A7C15ull);
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
double unit(uint64_t& s) { return ((splitmix64(s) >> 11) + 0.5) * (1.0 / 9007199254740992.0); }
}  // namespace

int pnn_net::bind(void* dev, size_t bytes) {
  if (!dev || (reinterpret_cast<uintptr_t>(dev) & 255)) return fail(PNN_EINVAL, "workspace must be 256-byte aligned");
  if (bytes < ws_bytes) return fail(PNN_ENOMEM, "workspace too small");
  ws = static_cast<char*>(dev);
  if (!stream) {
    // a library-owned blocking stream: ordered with the legacy default stream
    // and usable for CUDA-graph capture
    cudaError_t se = cudaStreamCreate(&stream);
    if (se != cudaSuccess) return cuda_check(se, "create stream");
    own_stream = true;
  }
  if (overlap_on && !s_hi) {
    int lo = 0, hi = 0, dev = 0, sms = 0;
    cudaError_t se = cudaDeviceGetStreamPriorityRange(&lo, &hi);
    if (se == cudaSuccess) se = cudaStreamCreateWithPriority(&s_hi, cudaStreamNonBlocking, hi);
    if (se == cudaSuccess) se = cudaStreamCreateWithPriority(&s_lo, cudaStreamNonBlocking, lo);
    for (cudaEvent_t* ev_ : {&fork_ev, &hi_done, &lo_done})
      if (se == cudaSuccess) se = cudaEventCreateWithFlags(ev_, cudaEventDisableTiming);
    if (se == cudaSuccess) se = cudaGetDevice(&dev);
    if (se == cudaSuccess) se = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (se != cudaSuccess) return cuda_check(se, "create overlap streams");
    lo_cap = std::max(1, sms - opt.overlap);
  }
  int r = build_tables();
  if (r) return r;
  if (host_tables.size() > tables_bytes) return fail(PNN_EINVAL, "internal: launch tables exceed their reservation");
  cudaError_t e = cudaMemcpy(ws + tables_off, host_tables.data(), host_tables.size(), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_check(e, "upload launch tables");
  // He-normal initialisation (std sqrt(2/fan_in)); BN gamma 1, beta 0; FC bias 0
  std::vector<float> theta(nparams), internal(nparams);
  uint64_t s = opt.seed * 0x2545F4914F6CDD1Dull + 1;
  for (const ParamT& p : params) {
    float* dst = theta.data() + p.off;
    if (p.kind == 0 || p.kind == 3) {
      const double fan_in = (double)p.n / p.dims[0];
      const double sd = std::sqrt(2.0 / fan_in);
      for (size_t i = 0; i < p.n; ++i) {
        const double u1 = unit(s), u2 = unit(s);
        dst[i] = (float)(sd * std::sqrt(-2.0 * std::log(u1)) * std::cos(6.283185307179586 * u2));
      }
    } else {
      for (size_t i = 0; i < p.n; ++i) dst[i] = p.kind == 1 ? 1.f : 0.f;
    }
  }
  for (const ParamT& p : params) to_internal(p, theta.data() + p.off, internal.data() + p.off);
  e = cudaMemcpy(ws + off_master, internal.data(), nparams * 4, cudaMemcpyHostToDevice);
  if (e == cudaSuccess && !opt.inference) e = cudaMemset(ws + off_grad, 0, nparams * 4);
  if (e == cudaSuccess && !opt.inference) e = cudaMemset(ws + off_mom, 0, nparams * 4);
  if (e == cudaSuccess && running_floats) {
    // running means 0, running variances 1
    std::vector<float> run(running_floats, 0.f);
    for (size_t i = 0; i < params.size(); ++i)
      if (params[i].kind == 1) std::fill(run.begin() + run_at[i] + params[i].n, run.begin() + run_at[i] + 2 * params[i].n, 1.f);
    e = cudaMemcpy(ws + off_running, run.data(), running_floats * 4, cudaMemcpyHostToDevice);
  }
  if (e == cudaSuccess) e = cudaMemset(ws + status_off, 0, 64);
  if (e == cudaSuccess && fin_cnt_bytes) e = cudaMemset(ws + off_fin_cnt, 0, fin_cnt_bytes);
  if (e == cudaSuccess && act_dt == DT_BF16)
    e = launch_copy_cast(P<float>(off_master), ws + off_shadow, DT_BF16, (int64_t)nparams, stream);
  if (e == cudaSuccess) e = refresh_wt();
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_check(e, "initialise parameters");
  for (auto& v : ev)
    if (!v) cudaEventCreate(&v);
  return PNN_OK;
}

// ====================================================================== C ABI
namespace {
thread_local std::string g_err;
int set_global(int code, const std::string& m) {
  g_err = m;
  return code;
}
}  // namespace

int pnn::set_last_error(int code, const char* msg) {
  g_err = msg ? msg : "";
  return code;
}

namespace {
#define NET_OR_FAIL(n) \
  if (!(n)) return set_global(PNN_EINVAL, "null handle");
#define BOUND_OR_FAIL(n)  \
  NET_OR_FAIL(n);         \
  if (!(n)->ws) return (n)->fail(PNN_ENOTBOUND, "no workspace bound");
#define TRAINING_OR_FAIL(n) \
  if ((n)->opt.inference) return (n)->fail(PNN_ESTATE, "an inference net runs pnn_infer only");
}  // namespace

extern "C" {

void pnn_default_options(pnn_options* o) {
  if (!o) return;
  memset(o, 0, sizeof *o);
  o->precision = PNN_BF16;
  o->correction = PNN_CORR_RESIDUAL;
  o->seed = 0;
  o->lr = 0.1f;
  o->momentum = 0.9f;
  o->weight_decay = 5e-4f;
  o->nesterov = 1;
  o->stream_fp32 = 1;
  o->conv_impl = 0;
  o->stream = nullptr;
  o->bn_momentum = 0.1f;
  o->inference = 0;
  o->overlap = 0;
  o->fuse_correction = 1;
}

int pnn_create(const pnn_desc* desc, const pnn_options* opts, pnn_net** out) {
  if (!desc || !out) return set_global(PNN_EINVAL, "null argument");
  *out = nullptr;
  pnn_net* n = new (std::nothrow) pnn_net();
  if (!n) return set_global(PNN_ENOMEM, "out of host memory");
  if (opts) n->opt = *opts;
  else pnn_default_options(&n->opt);
  if (n->opt.precision != PNN_BF16 && n->opt.precision != PNN_FP32_CHECK) {
    delete n;
    return set_global(PNN_EINVAL, "bad precision");
  }
  if (n->opt.correction != PNN_CORR_RESIDUAL && n->opt.correction != PNN_CORR_DELTA) {
    delete n;
    return set_global(PNN_EINVAL, "bad correction mode");
  }
  n->stream = static_cast<cudaStream_t>(n->opt.stream);
  int r = n->plan(desc);
  if (r) {
    set_global(r, n->err);
    delete n;
    return r;
  }
  // reserve the launch tables (sized by a dry build with a null base)
  n->ws = nullptr;
  n->build_tables();
  n->tables_bytes = align256(n->host_tables.size() + 4096);
  n->tables_off = n->alloc(n->tables_bytes);
  n->ws_bytes = n->cursor;
  n->host_tables.clear();
  *out = n;
  return PNN_OK;
}

int pnn_block_costs(const pnn_desc* desc, const pnn_options* opts, int32_t kind, double* out, int32_t n) {
  if (!desc || !out) return set_global(PNN_EINVAL, "null argument");
  if (kind != PNN_COST_FLOPS && kind != PNN_COST_BYTES) return set_global(PNN_EINVAL, "bad cost kind");
  if (n <= 0 || n != desc->n_body) return set_global(PNN_EINVAL, "n must equal the body length");
  // the untorn network: the whole body as one segment, no coarse network
  pnn_desc d = *desc;
  const int32_t whole = desc->n_body;
  d.segments = &whole;
  d.n_seg = 1;
  d.coarse = nullptr;
  d.coarse_len = nullptr;
  pnn_net* net = nullptr;
  int r = pnn_create(&d, opts, &net);
  if (r) return r;
  std::fill(out, out + n, 0.0);
  // forward ops of body layer i carry key[0] = i, their backward ops -i
  auto add = [&](const std::vector<int>& L, int sign) {
    for (int id : L) {
      const POp& o = net->ops[id];
      const int i = sign * o.key[0];
      if (i < 0 || i >= n) continue;
      double f = 0.0, b = 0.0;
      net->op_cost(o, f, b);
      out[i] += kind == PNN_COST_FLOPS ? f : b;
    }
  };
  add(net->fine_f[0], 1);
  add(net->fine_b[0], -1);
  pnn_destroy(net);
  return PNN_OK;
}

int pnn_partition(const double* cost, int32_t n, int32_t n_seg, int32_t* segments) {
  if (!cost || !segments) return set_global(PNN_EINVAL, "null argument");
  if (n_seg <= 0 || n < n_seg) return set_global(PNN_EINVAL, "need 1 <= n_seg <= n");
  if ((double)n_seg * n * n > 4e9) return set_global(PNN_EINVAL, "n_seg * n^2 above 4e9 (the exact cut's cost)");
  std::vector<double> S(n + 1, 0.0);
  for (int i = 0; i < n; ++i) {
    if (!(cost[i] >= 0.0) || !std::isfinite(cost[i])) return set_global(PNN_EINVAL, "costs must be finite and >= 0");
    S[i + 1] = S[i] + cost[i];
  }
  // best[i]: the smallest possible largest segment sum over partitions of the
  // first i layers into j segments (j = 1 .. n_seg, one row at a time)
  const double inf = std::numeric_limits<double>::infinity();
  std::vector<double> best(n + 1, inf), next(n + 1, inf);
  for (int i = 1; i <= n; ++i) best[i] = S[i];
  for (int j = 2; j <= n_seg; ++j) {
    std::fill(next.begin(), next.end(), inf);
    for (int i = j; i <= n; ++i)
      for (int k = j - 1; k < i; ++k) next[i] = std::min(next[i], std::max(best[k], S[i] - S[k]));
    best.swap(next);
  }
  const double T = best[n];
  // one optimal partition: every segment from the left takes as many layers as
  // the bound T allows while leaving one layer for each later segment
  int start = 0;
  for (int j = 0; j < n_seg; ++j) {
    const int later = n_seg - 1 - j;
    int end = start + 1;
    if (later == 0) end = n;
    else
      while (end < n - later && S[end + 1] - S[start] <= T) ++end;
    segments[j] = end - start;
    start = end;
  }
  return PNN_OK;
}

int pnn_workspace_bytes(const pnn_net* n, size_t* bytes) {
  NET_OR_FAIL(n);
  if (!bytes) return set_global(PNN_EINVAL, "null argument");
  *bytes = n->ws_bytes;
  return PNN_OK;
}

int pnn_bind_workspace(pnn_net* n, void* dev, size_t bytes) {
  NET_OR_FAIL(n);
  return n->bind(dev, bytes);
}

int pnn_forward(pnn_net* n, const float* x, const int32_t* labels, float* loss) {
  BOUND_OR_FAIL(n);
  TRAINING_OR_FAIL(n);
  if (!x || !labels) return n->fail(PNN_EINVAL, "null x or labels");
  n->x_dev = x;
  n->labels_dev = labels;
  int r = n->do_forward(true);
  if (r) return r;
  if (loss) {
    cudaError_t e = cudaMemcpyAsync(loss, n->ws + n->loss_off, 4, cudaMemcpyDeviceToDevice, n->stream);
    if (e != cudaSuccess) return n->cuda_check(e, "copy loss");
  }
  n->state = 1;
  return PNN_OK;
}

int pnn_backward(pnn_net* n) {
  BOUND_OR_FAIL(n);
  TRAINING_OR_FAIL(n);
  if (n->state != 1) return n->fail(PNN_ESTATE, "pnn_backward needs a preceding pnn_forward");
  int r = n->do_backward(true);
  if (r) return r;
  n->state = 2;
  return PNN_OK;
}

int pnn_sgd_step(pnn_net* n, float lr) {
  BOUND_OR_FAIL(n);
  TRAINING_OR_FAIL(n);
  if (n->state != 2) return n->fail(PNN_ESTATE, "pnn_sgd_step needs a preceding pnn_backward");
  int r = n->do_sgd(lr, true);
  if (r) return r;
  n->state = 0;
  return PNN_OK;
}

int pnn_train_step(pnn_net* n, const float* x, const int32_t* labels, float* loss) {
  BOUND_OR_FAIL(n);
  TRAINING_OR_FAIL(n);
  if (!x || !labels) return n->fail(PNN_EINVAL, "null x or labels");
  if (n->first_step) {
    // the first step initialises the momentum buffers; run it eagerly
    int r = pnn_forward(n, x, labels, loss);
    if (!r) r = pnn_backward(n);
    if (!r) r = pnn_sgd_step(n, 0.f);
    return r;
  }
  if (n->gexec && (x != n->g_x || labels != n->g_labels || loss != n->g_loss)) {
    cudaGraphExecDestroy(n->gexec);
    cudaGraphDestroy(n->graph);
    n->gexec = nullptr;
    n->graph = nullptr;
  }
  if (!n->gexec) {
    n->x_dev = x;
    n->labels_dev = labels;
    cudaError_t e = cudaStreamBeginCapture(n->stream, cudaStreamCaptureModeThreadLocal);
    if (e != cudaSuccess) return n->cuda_check(e, "begin capture");
    int r = n->do_forward(false);
    if (!r && loss) r = n->cuda_check(cudaMemcpyAsync(loss, n->ws + n->loss_off, 4, cudaMemcpyDeviceToDevice, n->stream), "copy loss");
    if (!r) r = n->do_backward(false);
    if (!r) r = n->do_sgd(0.f, false);
    cudaGraph_t g = nullptr;
    e = cudaStreamEndCapture(n->stream, &g);
    if (r) {
      if (g) cudaGraphDestroy(g);
      return r;
    }
    if (e != cudaSuccess) return n->cuda_check(e, "end capture");
    n->graph = g;
    e = cudaGraphInstantiate(&n->gexec, g, 0);
    if (e != cudaSuccess) return n->cuda_check(e, "instantiate graph");
    n->g_x = x;
    n->g_labels = labels;
    n->g_loss = loss;
  }
  n->state = 0;
  return n->cuda_check(cudaGraphLaunch(n->gexec, n->stream), "graph launch");
}

static void drop_phase_graphs(pnn_net* n) {
  for (auto& g : n->pgexec)
    if (g) {
      cudaGraphExecDestroy(g);
      g = nullptr;
    }
}

int pnn_time_phases(pnn_net* n, const float* x, const int32_t* labels, int32_t steps, float ms[10]) {
  BOUND_OR_FAIL(n);
  TRAINING_OR_FAIL(n);
  if (!x || !labels || !ms) return n->fail(PNN_EINVAL, "null argument");
  if (steps <= 0) return n->fail(PNN_EINVAL, "steps must be positive");
  if (n->prof) return n->fail(PNN_ESTATE, "phase timing needs profiling off");
  if (n->overlap_on) return n->fail(PNN_ESTATE, "phase timing needs the phases in sequence (opts.overlap = 0)");
  if (n->first_step) {
    int r = pnn_train_step(n, x, labels, nullptr);
    if (r) return r;
  }
  if (n->pgexec[0] && (x != n->px || labels != n->plabels)) drop_phase_graphs(n);
  n->x_dev = x;
  n->labels_dev = labels;
  if (!n->pgexec[0]) {
    for (int k = 0; k < 9; ++k) {
      cudaError_t e = cudaStreamBeginCapture(n->stream, cudaStreamCaptureModeThreadLocal);
      if (e != cudaSuccess) return n->cuda_check(e, "begin capture");
      int r = PNN_OK;
      if (k == 0) {
        e = launch_pack_input(x, n->ws + n->vals[n->x_in].off, n->vals[n->x_in].dt, n->B, n->in_c, n->in_h, n->in_w,
                              n->stream);
        r = e == cudaSuccess ? n->run_phase(0) : n->cuda_check(e, "pack input");
      } else if (k < 4) {
        r = n->run_phase(k);
      } else if (k == 6) {
        r = n->run_phase(6);
        if (!r) r = n->run_phase(7);
      } else if (k < 8) {
        r = n->run_phase(k == 7 ? 8 : k);
      } else {
        r = n->do_sgd(0.f, false);
        n->first_step = false;
      }
      cudaGraph_t g = nullptr;
      e = cudaStreamEndCapture(n->stream, &g);
      if (r || e != cudaSuccess) {
        if (g) cudaGraphDestroy(g);
        drop_phase_graphs(n);
        return r ? r : n->cuda_check(e, "end capture");
      }
      e = cudaGraphInstantiate(&n->pgexec[k], g, 0);
      cudaGraphDestroy(g);
      if (e != cudaSuccess) {
        drop_phase_graphs(n);
        return n->cuda_check(e, "instantiate graph");
      }
    }
    n->px = x;
    n->plabels = labels;
  }
  // events: ev[k] before phase graph k, ev[9] after the update
  cudaEvent_t ev[10];
  for (auto& e : ev)
    if (cudaEventCreate(&e) != cudaSuccess) return n->cuda_check(cudaGetLastError(), "event");
  double acc[9] = {};
  cudaError_t e = cudaSuccess;
  for (int s = 0; s < steps && e == cudaSuccess; ++s) {
    for (int k = 0; k < 9 && e == cudaSuccess; ++k) {
      e = cudaEventRecord(ev[k], n->stream);
      if (e == cudaSuccess) e = cudaGraphLaunch(n->pgexec[k], n->stream);
    }
    if (e == cudaSuccess) e = cudaEventRecord(ev[9], n->stream);
    if (e == cudaSuccess) e = cudaEventSynchronize(ev[9]);
    for (int k = 0; k < 9 && e == cudaSuccess; ++k) {
      float t = 0.f;
      e = cudaEventElapsedTime(&t, ev[k], ev[k + 1]);
      acc[k] += t;
    }
  }
  for (auto& v : ev) cudaEventDestroy(v);
  if (e != cudaSuccess) return n->cuda_check(e, "phase timing");
  n->state = 0;
  // graph order pre_f fine_f coarse_f post_f post_b coarse_b fine_b pre_b update
  // -> the order of pnn_get_timings: four forward, four backward (pre, fine,
  // coarse, post), update, total
  const int map[8] = {0, 1, 2, 3, 7, 6, 5, 4};
  float tot = 0.f;
  for (int i = 0; i < 8; ++i) {
    ms[i] = (float)(acc[map[i]] / steps);
    tot += ms[i];
  }
  ms[8] = (float)(acc[8] / steps);
  ms[9] = tot + ms[8];
  return pnn_sync(n);
}

int pnn_train_step_host(pnn_net* n, const float* x_host, const int32_t* labels_host, float* loss_host) {
  BOUND_OR_FAIL(n);
  TRAINING_OR_FAIL(n);
  if (!x_host || !labels_host) return n->fail(PNN_EINVAL, "null x or labels");
  const size_t xb = (size_t)n->B * n->in_c * n->in_h * n->in_w * 4;
  cudaError_t e = cudaMemcpyAsync(n->ws + n->x_stage, x_host, xb, cudaMemcpyHostToDevice, n->stream);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(n->ws + n->labels_stage, labels_host, (size_t)n->B * 4, cudaMemcpyHostToDevice, n->stream);
  if (e != cudaSuccess) return n->cuda_check(e, "copy inputs");
  int r = pnn_train_step(n, n->P<float>(n->x_stage), n->P<int32_t>(n->labels_stage), nullptr);
  if (r) return r;
  if (loss_host) {
    e = cudaMemcpyAsync(loss_host, n->ws + n->loss_off, 4, cudaMemcpyDeviceToHost, n->stream);
    if (e != cudaSuccess) return n->cuda_check(e, "copy loss");
  }
  return pnn_sync(n);
}

int pnn_sync(pnn_net* n) {
  BOUND_OR_FAIL(n);
  cudaError_t e = cudaStreamSynchronize(n->stream);
  if (e != cudaSuccess) return n->cuda_check(e, "synchronise");
  int32_t st = 0;
  e = cudaMemcpy(&st, n->ws + n->status_off, 4, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return n->cuda_check(e, "read status");
  if (st == 1) return n->fail(PNN_ENONFINITE, "label out of range");
  if (st == 2) return n->fail(PNN_ENONFINITE, "non-finite loss");
  if (st == 3) return n->fail(PNN_ETIMEOUT, "device wait timed out");
  return PNN_OK;
}

int pnn_running_stats_size(const pnn_net* n, size_t* out) {
  NET_OR_FAIL(n);
  if (!out) return set_global(PNN_EINVAL, "null argument");
  *out = n->running_floats;
  return PNN_OK;
}

int pnn_get_running_stats(pnn_net* n, float* host, size_t count) {
  BOUND_OR_FAIL(n);
  if ((!host && count) || count != n->running_floats) return n->fail(PNN_EINVAL, "length must equal pnn_running_stats_size");
  cudaError_t e = cudaStreamSynchronize(n->stream);
  if (e == cudaSuccess && count) e = cudaMemcpy(host, n->ws + n->off_running, count * 4, cudaMemcpyDeviceToHost);
  return n->cuda_check(e, "read running statistics");
}

int pnn_set_running_stats(pnn_net* n, const float* host, size_t count) {
  BOUND_OR_FAIL(n);
  if ((!host && count) || count != n->running_floats) return n->fail(PNN_EINVAL, "length must equal pnn_running_stats_size");
  cudaError_t e = cudaStreamSynchronize(n->stream);
  if (e == cudaSuccess && count) e = cudaMemcpy(n->ws + n->off_running, host, count * 4, cudaMemcpyHostToDevice);
  return n->cuda_check(e, "write running statistics");
}

int pnn_infer(pnn_net* n, const float* x, float* logits) {
  BOUND_OR_FAIL(n);
  if (!n->opt.inference) return n->fail(PNN_ESTATE, "pnn_infer needs a net created with opts.inference = 1");
  if (!x || !logits) return n->fail(PNN_EINVAL, "null x or logits");
  if (n->prof) {
    // profiling: eager launches, each bracketed by events
    n->x_dev = x;
    n->labels_dev = nullptr;
    int r = n->do_forward(true);
    const int nfc = (int)n->fc_width.size() - 1;
    if (!r)
      r = n->cuda_check(cudaMemcpyAsync(logits, n->ws + n->feat[nfc], (size_t)n->B * n->classes * 4,
                                        cudaMemcpyDeviceToDevice, n->stream),
                        "copy logits");
    return r;
  }
  if (n->igexec && (x != n->ix || logits != n->ilogits)) {
    cudaGraphExecDestroy(n->igexec);
    n->igexec = nullptr;
  }
  if (!n->igexec) {
    n->x_dev = x;
    n->labels_dev = nullptr;
    cudaError_t e = cudaStreamBeginCapture(n->stream, cudaStreamCaptureModeThreadLocal);
    if (e != cudaSuccess) return n->cuda_check(e, "begin capture");
    int r = n->do_forward(false);
    const int nfc = (int)n->fc_width.size() - 1;
    if (!r)
      r = n->cuda_check(cudaMemcpyAsync(logits, n->ws + n->feat[nfc], (size_t)n->B * n->classes * 4,
                                        cudaMemcpyDeviceToDevice, n->stream),
                        "copy logits");
    cudaGraph_t g = nullptr;
    e = cudaStreamEndCapture(n->stream, &g);
    if (r || e != cudaSuccess) {
      if (g) cudaGraphDestroy(g);
      return r ? r : n->cuda_check(e, "end capture");
    }
    e = cudaGraphInstantiate(&n->igexec, g, 0);
    cudaGraphDestroy(g);
    if (e != cudaSuccess) return n->cuda_check(e, "instantiate graph");
    n->ix = x;
    n->ilogits = logits;
  }
  return n->cuda_check(cudaGraphLaunch(n->igexec, n->stream), "graph launch");
}

void pnn_destroy(pnn_net* n) {
  if (!n) return;
  if (n->igexec) cudaGraphExecDestroy(n->igexec);
  if (n->gexec) cudaGraphExecDestroy(n->gexec);
  if (n->graph) cudaGraphDestroy(n->graph);
  drop_phase_graphs(n);
  for (auto& v : n->ev)
    if (v) cudaEventDestroy(v);
  for (auto& v : n->pev)
    if (v) cudaEventDestroy(v);
  if (n->own_stream && n->stream) cudaStreamDestroy(n->stream);
  for (cudaEvent_t v : {n->fork_ev, n->hi_done, n->lo_done})
    if (v) cudaEventDestroy(v);
  if (n->s_hi) cudaStreamDestroy(n->s_hi);
  if (n->s_lo) cudaStreamDestroy(n->s_lo);
  delete n;
}

int pnn_num_params(const pnn_net* n, size_t* out) {
  NET_OR_FAIL(n);
  if (!out) return set_global(PNN_EINVAL, "null argument");
  *out = n->nparams;
  return PNN_OK;
}

int pnn_num_param_tensors(const pnn_net* n, int32_t* out) {
  NET_OR_FAIL(n);
  if (!out) return set_global(PNN_EINVAL, "null argument");
  *out = (int32_t)n->params.size();
  return PNN_OK;
}

int pnn_param_tensor_info(const pnn_net* n, int32_t i, int32_t* kind, int32_t dims[4], size_t* offset) {
  NET_OR_FAIL(n);
  if (i < 0 || i >= (int32_t)n->params.size()) return set_global(PNN_EINVAL, "tensor index out of range");
  // i-th tensor in theta-bar order
  std::vector<int> order(n->params.size());
  for (size_t k = 0; k < order.size(); ++k) order[k] = (int)k;
  std::sort(order.begin(), order.end(), [&](int a, int b) { return n->params[a].off < n->params[b].off; });
  const ParamT& p = n->params[order[i]];
  if (kind) *kind = p.kind;
  if (dims)
    for (int k = 0; k < 4; ++k) dims[k] = p.dims[k];
  if (offset) *offset = p.off;
  return PNN_OK;
}

static int copy_params_out(pnn_net* n, size_t off, float* host, size_t count) {
  BOUND_OR_FAIL(n);
  if (!host || count != n->nparams) return n->fail(PNN_EINVAL, "length must equal pnn_num_params");
  std::vector<float> tmp(n->nparams);
  cudaError_t e = cudaStreamSynchronize(n->stream);
  if (e == cudaSuccess) e = cudaMemcpy(tmp.data(), n->ws + off, n->nparams * 4, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return n->cuda_check(e, "copy parameters out");
  for (const ParamT& p : n->params) to_external(p, tmp.data() + p.off, host + p.off);
  return PNN_OK;
}

int pnn_get_params(pnn_net* n, float* host, size_t count) { NET_OR_FAIL(n); return copy_params_out(n, n->off_master, host, count); }
int pnn_get_grads(pnn_net* n, float* host, size_t count) {
  NET_OR_FAIL(n);
  TRAINING_OR_FAIL(n);
  return copy_params_out(n, n->off_grad, host, count);
}
int pnn_get_momentum(pnn_net* n, float* host, size_t count) {
  NET_OR_FAIL(n);
  TRAINING_OR_FAIL(n);
  return copy_params_out(n, n->off_mom, host, count);
}

int pnn_set_params(pnn_net* n, const float* host, size_t count) {
  BOUND_OR_FAIL(n);
  if (!host || count != n->nparams) return n->fail(PNN_EINVAL, "length must equal pnn_num_params");
  std::vector<float> tmp(n->nparams);
  for (const ParamT& p : n->params) to_internal(p, host + p.off, tmp.data() + p.off);
  cudaError_t e = cudaStreamSynchronize(n->stream);
  if (e == cudaSuccess) e = cudaMemcpy(n->ws + n->off_master, tmp.data(), n->nparams * 4, cudaMemcpyHostToDevice);
  if (e == cudaSuccess && n->act_dt == DT_BF16)
    e = launch_copy_cast(n->P<float>(n->off_master), n->ws + n->off_shadow, DT_BF16, (int64_t)n->nparams, n->stream);
  if (e == cudaSuccess) e = n->refresh_wt();
  if (e == cudaSuccess) e = cudaStreamSynchronize(n->stream);
  return n->cuda_check(e, "set parameters");
}

static int tensor_value(const pnn_net* n, int which, int j, int* v, bool* grad) {
  const int N = n->N;
  *grad = false;
  *v = -1;
  const auto it = n->derived.find({which, j});
  if (it != n->derived.end()) {  // not stored: same shape as its first operand
    *v = std::get<0>(it->second);
    return PNN_OK;
  }
  switch (which) {
    case PNN_T_X: if (j >= 1 && j <= N) *v = n->xs[j - 1]; break;
    case PNN_T_Y: if (j >= 1 && j <= N) *v = n->ys[j - 1]; break;
    case PNN_T_R: if (j >= 1 && j < N) *v = n->rs[j - 1]; break;
    case PNN_T_RTILDE: if (j >= 1 && j <= N) *v = n->rts[j - 1]; break;
    case PNN_T_YTILDE: *v = n->ytilde; break;
    case PNN_T_D: if (j >= 1 && j <= N) { *v = n->rts[j - 1]; *grad = true; } break;
    case PNN_T_LOGITS: *v = -2; break;
  }
  return *v == -1 ? PNN_EINVAL : PNN_OK;
}

int pnn_tensor_size(const pnn_net* n, int32_t which, int32_t j, size_t* out) {
  NET_OR_FAIL(n);
  if (!out) return set_global(PNN_EINVAL, "null argument");
  int v; bool g;
  *out = 0;
  if (tensor_value(n, which, j, &v, &g)) return PNN_OK;
  if (v == -2) *out = (size_t)n->B * n->classes;
  else *out = (size_t)n->B * n->vals[v].C * n->vals[v].H * n->vals[v].W;
  return PNN_OK;
}

int pnn_get_tensor(pnn_net* n, int32_t which, int32_t j, float* host, size_t count) {
  BOUND_OR_FAIL(n);
  if (n->opt.inference && which != PNN_T_LOGITS)
    return n->fail(PNN_ESTATE, "an inference net keeps only the logits (its activations share buffers)");
  int v; bool g;
  if (tensor_value(n, which, j, &v, &g)) return n->fail(PNN_EINVAL, "no such tensor");
  size_t want;
  pnn_tensor_size(n, which, j, &want);
  if (!host || count != want) return n->fail(PNN_EINVAL, "length must equal pnn_tensor_size");
  // values the step does not store (the correction folded into conv
  // epilogues): y_j = r_j + x_{j+1}, rt_N = ytilde - y_N, from what it stores
  int a = -1, b = -1;
  float cb = 0.f;
  const auto it = n->derived.find({which, j});
  if (it != n->derived.end()) std::tie(a, b, cb) = it->second;
  if (a >= 0) {
    const Value& va = n->vals[a];
    std::vector<float> tmp(want);
    cudaError_t e = launch_export(make_src(*n, a), n->B, va.H, va.W, va.C, n->P<float>(n->export_off), n->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(n->stream);
    if (e == cudaSuccess) e = cudaMemcpy(host, n->ws + n->export_off, want * 4, cudaMemcpyDeviceToHost);
    if (e == cudaSuccess)
      e = launch_export(make_src(*n, b), n->B, va.H, va.W, va.C, n->P<float>(n->export_off), n->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(n->stream);
    if (e == cudaSuccess) e = cudaMemcpy(tmp.data(), n->ws + n->export_off, want * 4, cudaMemcpyDeviceToHost);
    if (e == cudaSuccess)
      for (size_t i = 0; i < want; ++i) host[i] += cb * tmp[i];
    return n->cuda_check(e, "export tensor");
  }
  cudaError_t e = cudaSuccess;
  if (v == -2) {
    const int nfc = (int)n->fc_width.size() - 1;
    e = cudaMemcpyAsync(n->ws + n->export_off, n->ws + n->feat[nfc], want * 4, cudaMemcpyDeviceToDevice, n->stream);
  } else if (which == PNN_T_RTILDE && n->N == 1) {
    // eq:correct with N = 1: rt_1 = r_1 = r_N = 0
    e = cudaMemsetAsync(n->ws + n->export_off, 0, want * 4, n->stream);
  } else {
    const Value& val = n->vals[v];
    Src s;
    if (g) {
      if (!val.need_grad) return n->fail(PNN_EINVAL, "no gradient for this tensor");
      s = Src{n->ws + n->gptr(v), nullptr, nullptr, DT_F32, 0};
    } else {
      s = make_src(*n, v);
    }
    e = launch_export(s, n->B, val.H, val.W, val.C, n->P<float>(n->export_off), n->stream);
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(n->stream);
  if (e == cudaSuccess) e = cudaMemcpy(host, n->ws + n->export_off, want * 4, cudaMemcpyDeviceToHost);
  return n->cuda_check(e, "export tensor");
}

int pnn_get_timings(pnn_net* n, float ms[10]) {
  BOUND_OR_FAIL(n);
  if (!ms) return n->fail(PNN_EINVAL, "null argument");
  cudaError_t e = cudaStreamSynchronize(n->stream);
  if (e != cudaSuccess) return n->cuda_check(e, "synchronise");
  auto el = [&](int a, int b) {
    float t = 0.f;
    if (cudaEventElapsedTime(&t, n->ev[a], n->ev[b]) != cudaSuccess) t = 0.f;
    return t;
  };
  ms[0] = el(0, 1); ms[1] = el(1, 2); ms[2] = el(2, 3); ms[3] = el(3, 4);
  ms[4] = el(8, 9); ms[5] = el(7, 8); ms[6] = el(6, 7); ms[7] = el(5, 6);
  ms[8] = el(10, 11);
  ms[9] = el(0, 4) + el(5, 9) + ms[8];
  cudaGetLastError();
  return PNN_OK;
}

int pnn_launch_counts(const pnn_net* n, int32_t counts[3]) {
  NET_OR_FAIL(n);
  if (!counts) return set_global(PNN_EINVAL, "null argument");
  int extra_head = 0;
  const int nfc = (int)n->fc_width.size() - 1;
  extra_head = 2 + nfc;  // gap, gemms, softmax
  counts[0] = n->counts[0] - 1 + extra_head + 1;  // + pack input
  counts[1] = n->counts[1] - 1 + 3 * nfc + (nfc - 1) + 1;
  counts[2] = n->counts[2];
  return PNN_OK;
}

int pnn_profile(pnn_net* n, int32_t enable) {
  BOUND_OR_FAIL(n);
  if (n->gexec) {
    cudaGraphExecDestroy(n->gexec);
    cudaGraphDestroy(n->graph);
    n->gexec = nullptr;
    n->graph = nullptr;
  }
  drop_phase_graphs(n);
  n->prof = enable != 0;
  n->pnext = 0;
  n->pfold = 0;
  for (int k = 0; k <= K_NKINDS; ++k) { n->kms[k] = 0; n->kflops[k] = 0; n->kbytes[k] = 0; n->klaunch[k] = 0; }
  return PNN_OK;
}

int pnn_profile_read(pnn_net* n, int32_t kind, double* ms, int64_t* launches, double* flops, double* bytes) {
  BOUND_OR_FAIL(n);
  if (kind < 0 || kind >= K_NKINDS) return n->fail(PNN_EINVAL, "bad kernel kind");
  cudaError_t e = cudaStreamSynchronize(n->stream);
  if (e != cudaSuccess) return n->cuda_check(e, "synchronise");
  // fold launches recorded since the last read into the per-kind totals
  for (size_t i = n->pfold; i + 1 < n->pnext; i += 2) {
    float t = 0.f;
    cudaEventElapsedTime(&t, n->pev[i], n->pev[i + 1]);
    const Launch& L = *n->plaunch[i / 2];
    n->kms[L.kind] += t;
    n->kflops[L.kind] += L.flops;
    n->kbytes[L.kind] += L.bytes;
    n->klaunch[L.kind] += 1;
  }
  n->pfold = n->pnext;
  if (ms) *ms = n->kms[kind];
  if (launches) *launches = n->klaunch[kind];
  if (flops) *flops = n->kflops[kind];
  if (bytes) *bytes = n->kbytes[kind];
  return PNN_OK;
}

int pnn_profile_trace(pnn_net* n, int32_t max, pnn_trace* out, int32_t* count) {
  BOUND_OR_FAIL(n);
  if (max < 0 || (max > 0 && !out) || !count) return n->fail(PNN_EINVAL, "bad trace buffer");
  cudaError_t e = cudaStreamSynchronize(n->stream);
  if (e != cudaSuccess) return n->cuda_check(e, "synchronise");
  const int32_t have = (int32_t)(n->pnext / 2);
  for (int32_t i = 0; i < std::min(have, max); ++i) {
    const Launch& L = *n->plaunch[i];
    pnn_trace& r = out[i];
    float t = 0.f;
    cudaEventElapsedTime(&t, n->pev[2 * i], n->pev[2 * i + 1]);
    r.kind = L.kind; r.variant = L.variant + (L.wide ? 1 : (L.op > 0 ? 2 : 0)); r.phase = L.phase; r.instances = L.count;
    r.tiles = L.total;
    for (int j = 0; j < 6; ++j) r.shape[j] = L.shape[j];
    r.block = L.block;
    r.ms = t; r.flops = L.flops; r.bytes = L.bytes;
  }
  *count = have;
  return PNN_OK;
}

const char* pnn_kernel_kind_name(int32_t kind) {
  return (kind >= 0 && kind < K_NKINDS) ? kKindName[kind] : nullptr;
}

int32_t pnn_num_kernel_kinds(void) { return K_NKINDS; }

uint64_t pnn_debug_word(void) { return conv_tc_debug_word(); }

const char* pnn_last_error(const pnn_net* n) { return n ? n->err.c_str() : g_err.c_str(); }

const char* pnn_status_string(int s) {
  switch (s) {
    case PNN_OK: return "ok";
    case PNN_EINVAL: return "invalid argument";
    case PNN_ENOMEM: return "workspace too small";
    case PNN_ECUDA: return "CUDA error";
    case PNN_ESTATE: return "call out of order";
    case PNN_ETIMEOUT: return "device wait timed out";
    case PNN_ENONFINITE: return "non-finite loss or bad label";
    case PNN_ENOTBOUND: return "no workspace bound";
  }
  return "unknown status";
}

}  // extern "C"
