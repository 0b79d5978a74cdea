// One grouped convolution on caller buffers (pnn_conv_run): the forward, data
// gradient and weight gradient of Section 3.2's layers through the same
// tensor-core kernels and epilogues a training step launches, with the same
// tile rules, tensor maps and reductions, so that each kernel can be checked
// alone.  Also the tensor-map encoder both this file and the training
// runtime use.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstring>
#include <mutex>
#include <vector>

#include "../../include/pnn.h"
#include "pnn_internal.h"

namespace pnn {

int encode_tensor_map_2d(void* map, const void* base, bool bf16, int64_t inner, int64_t rows, int box_inner,
                         int box_rows, int swz, const char** why) {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  static std::once_flag once;
  std::call_once(once, []() {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    const cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e == cudaSuccess && q == cudaDriverEntryPointSuccess && fn)
      encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  if (!encode) {
    *why = "cuTensorMapEncodeTiled is not available from the driver";
    return 1;
  }
  const int esz = bf16 ? 2 : 4;
  const cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)rows};
  const cuuint64_t pitch[1] = {(cuuint64_t)inner * esz};
  const cuuint32_t box[2] = {(cuuint32_t)box_inner, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = encode(reinterpret_cast<CUtensorMap*>(map),
                            bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2,
                            const_cast<void*>(base), dims, pitch, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                            swz == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                            : swz == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                            : swz == 32 ? CU_TENSOR_MAP_SWIZZLE_32B
                                        : CU_TENSOR_MAP_SWIZZLE_NONE,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    *why = "cuTensorMapEncodeTiled rejected a conv operand map";
    return 1;
  }
  return 0;
}

namespace {

size_t al256(size_t x) { return (x + 255) & ~(size_t)255; }
int cdv(int64_t a, int64_t b) { return (int)((a + b - 1) / b); }

// The plan of one pnn_conv_run call: per instance its tile grid and the
// byte offsets of its scratch in the workspace; the launch-wide kernel
// parameters.
struct InstPlan {
  int P = 0, Q = 0, pad = 0, mtiles = 0, ntiles = 0, splits = 1, pix_per_split = 0, rows = 0;
  size_t wt = 0, part = 0, stats = 0, fscr = 0, fcnt = 0, gam = 0, bet = 0, scl = 0, shf = 0, coef = 0;
  size_t maps = 0;
  int stat_tiles = 0;
  bool bn = false;    // forward statistics / data-gradient BN sums requested
  bool halo = false;  // TMA-fed 3x3 forward / data gradient with halo tiles
};
struct Plan {
  int variant = 0;
  int bnmax = 16, raw = 0, op = 0, wide = 0;
  int total = 0;
  size_t tab = 0, ts = 0, status = 0, aux_tab = 0, aux_ts = 0, fin_tab = 0, fin_ts = 0, red_tab = 0, red_ts = 0;
  size_t bytes = 0, init_bytes = 0;  // init_bytes: the prefix copied from the host
  std::vector<InstPlan> in;
};

int check_args(int mode, int impl, int n, const pnn_conv_args* a) {
  if (mode < 0 || mode > 2 || impl < 0 || impl > 3 || n <= 0 || n > 4096 || !a)
    return set_last_error(PNN_EINVAL, "pnn_conv_run: bad mode, impl or instance count");
  for (int i = 0; i < n; ++i) {
    const pnn_conv_args& g = a[i];
    if (g.batch <= 0 || g.h <= 0 || g.w <= 0 || g.c <= 0 || g.k <= 0 || (g.ksize != 1 && g.ksize != 3) ||
        (g.stride != 1 && g.stride != 2))
      return set_last_error(PNN_EINVAL, "pnn_conv_run: bad geometry");
    if (g.c % 8 || g.k % 8) return set_last_error(PNN_EINVAL, "pnn_conv_run: c and k must be multiples of 8");
    if ((int64_t)g.batch * g.h * g.w > 0x7fffffffLL / std::max(g.c, g.k))
      return set_last_error(PNN_EINVAL, "pnn_conv_run: tensor too large");
    if (!g.wt) return set_last_error(PNN_EINVAL, "pnn_conv_run: null weights");
    if (mode == 0 && (!g.x || !g.y)) return set_last_error(PNN_EINVAL, "pnn_conv_run: forward needs x and y");
    if (mode == 0 && (!g.y_mean) != (!g.y_rstd))
      return set_last_error(PNN_EINVAL, "pnn_conv_run: y_mean and y_rstd go together");
    if (mode == 1 && (!g.dy || !g.dx)) return set_last_error(PNN_EINVAL, "pnn_conv_run: data gradient needs dy and dx");
    if (mode == 1 && g.bn_mean && (!g.x || !g.bn_rstd || !g.bn_scale || !g.bn_shift || !g.dgamma || !g.dbeta))
      return set_last_error(PNN_EINVAL, "pnn_conv_run: BN-backward sums need x, bn_scale/shift/mean/rstd, dgamma, dbeta");
    if (mode == 2 && (!g.x || !g.dy || !g.dw)) return set_last_error(PNN_EINVAL, "pnn_conv_run: weight gradient needs x, dy, dw");
    if ((!g.bn_scale) != (!g.bn_shift)) return set_last_error(PNN_EINVAL, "pnn_conv_run: bn_scale and bn_shift go together");
    if ((g.x_dtype != PNN_DT_F32 && g.x_dtype != PNN_DT_BF16) || (g.y_dtype != PNN_DT_F32 && g.y_dtype != PNN_DT_BF16) ||
        (g.res_dtype != PNN_DT_F32 && g.res_dtype != PNN_DT_BF16))
      return set_last_error(PNN_EINVAL, "pnn_conv_run: bad dtype");
    if (g.bn_scale && std::max(g.c, g.k) > 512)
      return set_last_error(PNN_EINVAL, "pnn_conv_run: at most 512 channels with a BN input transform");
  }
  return PNN_OK;
}

// which kernel every instance can take: 1 TMA-fed, 0 thread-gathered
bool tma_ok(int mode, const pnn_conv_args& g) {
  const int pad = g.ksize / 2;
  if (mode == 0) return tma_shape_ok(g.ksize, g.stride, pad, g.c);
  if (mode == 1) return tma_shape_ok(g.ksize, g.stride, pad, g.k);
  return tma_wgrad_ok(g.ksize, g.stride, pad, g.c, g.k, g.w, g.x_dtype == PNN_DT_BF16);
}

// whether instance g of a TMA-fed forward / data-gradient launch takes halo tiles
bool halo_inst(int mode, const pnn_conv_args& g) {
  if (mode == 2) return false;
  const int ncols = mode == 1 ? g.c : g.k, ch = mode == 1 ? g.k : g.c;
  const int bn = ncols <= tc_ntile_cols(mode, 1) ? ((ncols + 15) & ~15) : tc_ntile_cols(mode, 1);
  return halo_ok(g.ksize, g.stride, g.ksize / 2, g.h, g.w, ch) && conv_halo_fits(mode, g.w, ch, bn);
}

int make_plan(int mode, int impl, int n, const pnn_conv_args* a, Plan& pl) {
  int r = check_args(mode, impl, n, a);
  if (r) return r;
  // (an instance with halo tiles needs no per-tap boxes)
  bool all_tma = true, all_tap = true;
  for (int i = 0; i < n; ++i) {
    all_tap = all_tap && tma_ok(mode, a[i]);
    all_tma = all_tma && (tma_ok(mode, a[i]) || halo_inst(mode, a[i]));
  }
  if ((impl == 1 && !all_tma) || (impl == 3 && !all_tap))
    return set_last_error(PNN_EINVAL, "pnn_conv_run: the TMA-fed kernel does not take this shape");
  // the training step's rule: TMA-fed where the shape allows (the forward only
  // for at least 64 output channels or with halo tiles)
  bool auto_tma = all_tma;
  if (mode == 0)
    for (int i = 0; i < n; ++i) auto_tma = auto_tma && ((a[i].k >= 64 && tma_ok(mode, a[i])) || halo_inst(mode, a[i]));
  pl.variant = (impl == 1 || impl == 3) ? 1 : (impl == 2 ? 0 : (auto_tma ? 1 : 0));
  size_t cur = 0;
  auto take = [&](size_t b) { size_t o = cur; cur = al256(cur + b); return o; };
  pl.tab = take((size_t)n * sizeof(ConvDesc));
  pl.ts = take((size_t)(n + 1) * sizeof(int));
  pl.status = take(64);
  pl.aux_tab = take((size_t)n * std::max(sizeof(WtDesc), std::max(sizeof(WReduceDesc), sizeof(BnBwdDesc))));
  pl.aux_ts = take((size_t)(n + 1) * sizeof(int));
  pl.fin_tab = take((size_t)n * std::max(sizeof(BnFinDesc), sizeof(BnBwdDesc)));
  pl.fin_ts = take((size_t)(n + 1) * sizeof(int));
  pl.red_tab = take((size_t)n * sizeof(BnBwdDesc));
  pl.red_ts = take((size_t)(n + 1) * sizeof(int));
  pl.in.resize(n);
  const int sms = device_sm_count();
  pl.total = 0;
  pl.bnmax = 16;
  pl.raw = 0;
  int esz = 2;
  // pass 1: tile grids and the small regions that start from host values
  // (tensor maps, gamma / beta, finalize counters); pass 2: device scratch
  for (int i = 0; i < n; ++i) {
    const pnn_conv_args& g = a[i];
    InstPlan& ip = pl.in[i];
    ip.pad = g.ksize / 2;
    ip.P = (g.h + 2 * ip.pad - g.ksize) / g.stride + 1;
    ip.Q = (g.w + 2 * ip.pad - g.ksize) / g.stride + 1;
    if (ip.P <= 0 || ip.Q <= 0) return set_last_error(PNN_EINVAL, "pnn_conv_run: empty output");
    const int64_t Mout = (int64_t)g.batch * ip.P * ip.Q, Min = (int64_t)g.batch * g.h * g.w;
    const int rsc = g.ksize * g.ksize * g.c;
    const int ncols = mode == 1 ? g.c : g.k;
    ip.ntiles = mode == 2 ? cdv(g.k, 256) : cdv(ncols, tc_ntile_cols(mode, pl.variant));
    pl.bnmax = std::max(pl.bnmax, ip.ntiles == 1 ? ((ncols + 15) & ~15) : tc_ntile_cols(mode, pl.variant));
    if (mode == 0) {
      ip.mtiles = cdv(Mout, kTcBM);
      if (g.x_dtype == PNN_DT_F32) esz = 4;
      ip.bn = g.y_mean != nullptr;
      if (ip.bn) {
        ip.stat_tiles = ip.mtiles;
        ip.fcnt = take((size_t)cdv(g.k, 32) * 4);
        ip.gam = take((size_t)g.k * 4);
        ip.bet = take((size_t)g.k * 4);
      }
      pl.total += ip.mtiles * ip.ntiles;
    } else if (mode == 1) {
      ip.mtiles = cdv(Min, kTcBM);
      esz = 4;
      ip.bn = g.bn_mean != nullptr;
      if (ip.bn) {
        // the fused sums use 128-row tiles; the separate reduction its own
        ip.stat_tiles = std::max(ip.mtiles, cdv(Min, bnb_rows_per_tile(g.c)));
        ip.fcnt = take((size_t)cdv(g.c, 32) * 4);
        ip.gam = take((size_t)g.c * 4);
      }
      pl.total += ip.mtiles * ip.ntiles;
    } else {
      ip.rows = tc_tile_rows(2, pl.variant, g.c);
      ip.mtiles = cdv(rsc, ip.rows);
      const int base = ip.mtiles * ip.ntiles;
      int splits = std::max(1, std::min(cdv(Mout, 256), cdv(2 * (int64_t)sms, base)));
      ip.pix_per_split = cdv(cdv(Mout, splits), 64) * 64;
      ip.splits = cdv(Mout, ip.pix_per_split);
      if (pl.variant == 1) {
        const WgBoxes b = wg_boxes(g.c, g.k, g.w, ip.pad, g.x_dtype == PNN_DT_BF16);
        pl.raw = std::max(pl.raw, wg_raw_bytes(b));
      }
      pl.total += base * ip.splits;
    }
    ip.halo = pl.variant == 1 && impl != 3 && halo_inst(mode, g);
    if (pl.variant == 1) ip.maps = take(4 * 128);
  }
  pl.init_bytes = cur;
  for (int i = 0; i < n; ++i) {
    const pnn_conv_args& g = a[i];
    InstPlan& ip = pl.in[i];
    const int rsc = g.ksize * g.ksize * g.c;
    if (mode == 0 && ip.bn) {
      ip.stats = take((size_t)ip.stat_tiles * g.k * 8);
      ip.fscr = take((size_t)cdv(ip.stat_tiles, kFinTilesPerCta) * g.k * 16);
      ip.scl = take((size_t)g.k * 4);
      ip.shf = take((size_t)g.k * 4);
    } else if (mode == 1) {
      ip.wt = take((size_t)g.k * rsc * 2);
      if (ip.bn) {
        ip.stats = take((size_t)ip.stat_tiles * g.c * 8);
        ip.fscr = take((size_t)cdv(ip.stat_tiles, kFinTilesPerCta) * g.c * 16);
        ip.coef = take((size_t)g.c * 12);
      }
    } else if (mode == 2) {
      ip.part = take((size_t)ip.splits * g.k * rsc * 4);
    }
  }
  if (pl.variant == 1 && mode != 2) {
    // per instance: one tap box per k-step, or (halo tiles) one halo box per tile
    pl.raw = 1024;
    for (int i = 0; i < n; ++i) {
      const pnn_conv_args& g = a[i];
      const int ch = mode == 1 ? g.k : g.c, ncols = mode == 1 ? g.c : g.k;
      if (pl.in[i].halo) {
        const int bn = pl.in[i].ntiles == 1 ? ((ncols + 15) & ~15) : tc_ntile_cols(mode, 1);
        pl.raw = std::max(pl.raw, halo_raw_bytes(g.w, ch, esz));
        pl.op = std::max(pl.op, halo_op_bytes(g.w, ch, bn));
      } else {
        pl.raw = std::max(pl.raw, kTcBM * 64 * esz);
      }
    }
    if (pl.op > 0) pl.op = std::max(pl.op, conv_tma_op_bytes(mode, pl.bnmax));
  }
  // the training step's rule: the wide-epilogue variant when every tile is
  // one k-step
  pl.wide = pl.variant == 1 && mode != 2;
  for (int i = 0; i < n; ++i)
    if (a[i].ksize * a[i].ksize * (mode == 0 ? a[i].c : a[i].k) > 64) pl.wide = 0;
  pl.bytes = cur;
  return PNN_OK;
}

}  // namespace
}  // namespace pnn

using namespace pnn;

extern "C" int pnn_conv_workspace_bytes(int32_t mode, int32_t impl, int32_t n, const pnn_conv_args* args, size_t* bytes) {
  if (!bytes) return set_last_error(PNN_EINVAL, "pnn_conv_workspace_bytes: null output");
  Plan pl;
  const int r = make_plan(mode, impl, n, args, pl);
  if (r) return r;
  *bytes = pl.bytes;
  return PNN_OK;
}

namespace {
int conv_run(int32_t mode, int32_t impl, int32_t n, const pnn_conv_args* a, void* workspace, size_t workspace_bytes,
             void* stream, int repeat, float* ms_out) {
  Plan pl;
  int r = make_plan(mode, impl, n, a, pl);
  if (r) return r;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255))
    return set_last_error(PNN_EINVAL, "pnn_conv_run: workspace must be a 256-byte aligned device pointer");
  if (workspace_bytes < pl.bytes) return set_last_error(PNN_ENOMEM, "pnn_conv_run: workspace too small");
  char* ws = static_cast<char*>(workspace);
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  // host images of every table, copied into the workspace before the launches
  std::vector<uint8_t> img(pl.init_bytes, 0);
  auto at = [&](size_t off) { return img.data() + off; };
  std::vector<ConvDesc> cds(n);
  std::vector<int> ts(n + 1, 0);
  std::vector<WtDesc> wts;
  std::vector<WReduceDesc> wrs;
  std::vector<BnFinDesc> fins;
  std::vector<BnBwdDesc> bfins, breds;
  std::vector<int> aux_ts(1, 0), fin_ts(1, 0), red_ts(1, 0);
  int32_t* status = reinterpret_cast<int32_t*>(ws + pl.status);
  for (int i = 0; i < n; ++i) {
    const pnn_conv_args& g = a[i];
    const InstPlan& ip = pl.in[i];
    ConvDesc& c = cds[i];
    c = ConvDesc{};
    c.x = Src{g.x, g.bn_scale, g.bn_shift, g.x_dtype, g.bn_scale ? g.relu : 0};
    c.w = g.wt;
    c.w_dt = DT_BF16;
    c.B = g.batch; c.H = g.h; c.W = g.w; c.C = g.c; c.P = ip.P; c.Q = ip.Q; c.K = g.k;
    c.R = g.ksize; c.S = g.ksize; c.stride = g.stride; c.pad = ip.pad;
    c.mtiles = ip.mtiles; c.ntiles = ip.ntiles;
    c.ntile_w = tc_ntile_cols(mode, pl.variant);
    c.mtile_rows = tc_tile_rows(mode, pl.variant, g.c);
    c.op_bf16 = 1;
    const int64_t Mout = (int64_t)g.batch * ip.P * ip.Q, Min = (int64_t)g.batch * g.h * g.w;
    const int rsc = g.ksize * g.ksize * g.c;
    if (mode == 0) {
      c.y = g.y; c.y_dt = g.y_dtype;
      if (g.res) { c.res = g.res; c.res_dt = g.res_dtype; }
      if (ip.bn) c.stats = reinterpret_cast<float*>(ws + ip.stats);
    } else if (mode == 1) {
      c.w = ws + ip.wt;  // the transposed bf16 weights Wt[c][r][s][k]
      c.dy = g.dy;
      c.dx = g.dx;
      c.accumulate = g.accumulate ? 1 : 0;
      WtDesc w{};
      w.src = g.wt; w.dst = ws + ip.wt; w.K = g.k; w.RS = g.ksize * g.ksize; w.C = g.c; w.n = (int64_t)g.k * rsc;
      wts.push_back(w);
      aux_ts.push_back(aux_ts.back() + cdv(w.n, 256));
    } else {
      c.dy = g.dy;
      c.dw_part = reinterpret_cast<float*>(ws + ip.part);
      c.splits = ip.splits;
      c.pix_per_split = ip.pix_per_split;
      WReduceDesc w{};
      w.part = c.dw_part; w.dw = g.dw; w.splits = ip.splits; w.accumulate = 0; w.n = (int64_t)g.k * rsc;
      w.tiles = cdv(w.n, 32); w.transposed = 1; w.kout = g.k; w.rsc = rsc;
      wrs.push_back(w);
      aux_ts.push_back(aux_ts.back() + w.tiles);
    }
    if (pl.variant == 1) {
      const char* why = nullptr;
      uint8_t* m = at(ip.maps);
      int e = 0;
      if (mode == 0) {
        const int bn = ip.ntiles == 1 ? ((g.k + 15) & ~15) : tc_ntile_cols(0, 1);
        e = encode_tensor_map_2d(m, g.x, g.x_dtype == PNN_DT_BF16, g.c, Min, std::min(g.c, 64), kTcBM, 0, &why);
        if (!e) e = encode_tensor_map_2d(m + 128, g.wt, true, rsc, g.k, 64, bn, 128, &why);
        if (!e) e = encode_tensor_map_2d(m + 256, g.y, g.y_dtype == PNN_DT_BF16, g.k, Mout, 16, 32,
                                         g.y_dtype == PNN_DT_BF16 ? 32 : 64, &why);
        if (!e && ip.halo)
          e = encode_tensor_map_2d(m + 384, g.x, g.x_dtype == PNN_DT_BF16, g.c, Min, g.c, halo_rows(g.w), 0, &why);
      } else if (mode == 1) {
        const int bn = ip.ntiles == 1 ? ((g.c + 15) & ~15) : tc_ntile_cols(1, 1);
        e = encode_tensor_map_2d(m, g.dy, false, g.k, Mout, std::min(g.k, 64), kTcBM, 0, &why);
        if (!e) e = encode_tensor_map_2d(m + 128, ws + ip.wt, true, g.ksize * g.ksize * g.k, g.c, 64, bn, 128, &why);
        if (!e) e = encode_tensor_map_2d(m + 256, g.dx, false, g.c, Min, 16, 32, 64, &why);
        if (!e && ip.halo) e = encode_tensor_map_2d(m + 384, g.dy, false, g.k, Mout, g.k, halo_rows(g.w), 0, &why);
      } else {
        const WgBoxes bx = wg_boxes(g.c, g.k, g.w, ip.pad, g.x_dtype == PNN_DT_BF16);
        e = encode_tensor_map_2d(m, g.x, g.x_dtype == PNN_DT_BF16, g.c, Min, bx.cwx, bx.hrows, 0, &why);
        if (!e) e = encode_tensor_map_2d(m + 128, g.dy, false, g.k, Mout, g.k, 64, 0, &why);
      }
      if (e) return set_last_error(PNN_ECUDA, why);
      c.tma_a = ws + ip.maps;
      c.tma_b = ws + ip.maps + 128;
      c.tma_y = mode == 2 ? nullptr : ws + ip.maps + 256;
      c.tma_h = ip.halo ? ws + ip.maps + 384 : nullptr;
    }
    if (ip.bn && mode == 0) {
      // forward statistics: the epilogue's per-tile partials, then the
      // finalize kernel with gamma = 1, beta = 0 (mean and rstd out)
      float* gam = reinterpret_cast<float*>(at(ip.gam));
      for (int k = 0; k < g.k; ++k) gam[k] = 1.f;
      BnFinDesc f{};
      f.part = c.stats; f.tiles = ip.stat_tiles; f.C = g.k; f.count = Mout; f.rows_per_tile = kTcBM;
      f.gamma = reinterpret_cast<const float*>(ws + ip.gam); f.beta = reinterpret_cast<const float*>(ws + ip.bet);
      f.mean = g.y_mean; f.rstd = g.y_rstd;
      f.scale = reinterpret_cast<float*>(ws + ip.scl); f.shift = reinterpret_cast<float*>(ws + ip.shf);
      f.momentum = 0.f; f.eval = 0;
      f.scratch = reinterpret_cast<double*>(ws + ip.fscr); f.counter = reinterpret_cast<int32_t*>(ws + ip.fcnt);
      f.cgroups = cdv(g.k, 32);
      f.nchunk = cdv(std::max(ip.stat_tiles, 1), kFinTilesPerCta);
      fins.push_back(f);
      fin_ts.push_back(fin_ts.back() + f.cgroups * f.nchunk);
    }
    if (ip.bn && mode == 1) {
      float* gam = reinterpret_cast<float*>(at(ip.gam));
      for (int k = 0; k < g.c; ++k) gam[k] = 1.f;
      BnBwdDesc b{};
      b.da = g.dx;
      b.h = g.x; b.h_dt = g.x_dtype;
      b.mean = g.bn_mean; b.rstd = g.bn_rstd; b.scale = g.bn_scale; b.shift = g.bn_shift;
      b.gamma = reinterpret_cast<const float*>(ws + ip.gam);
      b.relu = g.relu ? 1 : 0;
      b.part = reinterpret_cast<float*>(ws + ip.stats);
      b.dgamma = g.dgamma; b.dbeta = g.dbeta;
      b.coef = reinterpret_cast<float*>(ws + ip.coef);
      b.M = Min; b.C = g.c;
      b.rows_per_tile = bnb_rows_per_tile(g.c);
      b.scratch = reinterpret_cast<double*>(ws + ip.fscr); b.counter = reinterpret_cast<int32_t*>(ws + ip.fcnt);
      b.cgroups = cdv(g.c, 32);
      // the TMA-fed data gradient forms the sums of its 128-row tiles in its
      // epilogue when it writes the whole gradient; otherwise the separate
      // reduction kernel runs over its own row tiles
      const bool fused = pl.variant == 1 && !g.accumulate && g.c % 16 == 0;
      if (fused) {
        c.bn_mean = g.bn_mean; c.bn_rstd = g.bn_rstd; c.bnb_part = b.part;
        b.tiles = ip.mtiles;
      } else {
        if (g.c % 8 != 0 || g.c > 2048) return set_last_error(PNN_EINVAL, "pnn_conv_run: BN sums need c % 8 == 0");
        b.tiles = cdv(Min, bnb_rows_per_tile(g.c));
        breds.push_back(b);
        red_ts.push_back(red_ts.back() + b.tiles);
      }
      b.nchunk = cdv(std::max(b.tiles, 1), kFinTilesPerCta);
      b.accumulate = 0;
      bfins.push_back(b);
      fin_ts.push_back(fin_ts.back() + b.cgroups * b.nchunk);
    }
    ts[i + 1] = ts[i] + (mode == 2 ? ip.mtiles * ip.ntiles * ip.splits : ip.mtiles * ip.ntiles);
  }
  memcpy(at(pl.tab), cds.data(), cds.size() * sizeof(ConvDesc));
  memcpy(at(pl.ts), ts.data(), ts.size() * sizeof(int));
  if (!wts.empty()) memcpy(at(pl.aux_tab), wts.data(), wts.size() * sizeof(WtDesc));
  if (!wrs.empty()) memcpy(at(pl.aux_tab), wrs.data(), wrs.size() * sizeof(WReduceDesc));
  memcpy(at(pl.aux_ts), aux_ts.data(), aux_ts.size() * sizeof(int));
  if (!fins.empty()) memcpy(at(pl.fin_tab), fins.data(), fins.size() * sizeof(BnFinDesc));
  if (!bfins.empty()) memcpy(at(pl.fin_tab), bfins.data(), bfins.size() * sizeof(BnBwdDesc));
  memcpy(at(pl.fin_ts), fin_ts.data(), fin_ts.size() * sizeof(int));
  if (!breds.empty()) memcpy(at(pl.red_tab), breds.data(), breds.size() * sizeof(BnBwdDesc));
  memcpy(at(pl.red_ts), red_ts.data(), red_ts.size() * sizeof(int));
  // (the image zero-fills the status word, the finalize counters and beta)
  cudaError_t e = cudaMemcpyAsync(ws, img.data(), pl.init_bytes, cudaMemcpyHostToDevice, st);
  const auto* tab = reinterpret_cast<const ConvDesc*>(ws + pl.tab);
  const int* tsd = reinterpret_cast<const int*>(ws + pl.ts);
  const int* auxts = reinterpret_cast<const int*>(ws + pl.aux_ts);
  if (e == cudaSuccess && mode == 1)
    e = launch_wtrans(reinterpret_cast<const WtDesc*>(ws + pl.aux_tab), auxts, n, aux_ts.back(), st);
  auto conv_launch = [&]() {
    if (pl.variant == 1)
      return launch_conv_tma(mode, pl.wide, tab, tsd, n, pl.total, pl.bnmax, pl.raw, pl.op, status, st);
    if (mode == 0) return launch_conv_fwd_tc(tab, tsd, n, pl.total, pl.bnmax, status, st);
    if (mode == 1) return launch_conv_dgrad_tc(tab, tsd, n, pl.total, pl.bnmax, status, st);
    return launch_conv_wgrad_tc(tab, tsd, n, pl.total, pl.bnmax, status, st);
  };
  if (e == cudaSuccess) e = conv_launch();
  if (e == cudaSuccess && repeat > 0) {
    // device time of the conv kernel alone: `repeat` further launches (each
    // rewrites what the first wrote) between two events on the stream
    cudaEvent_t t0 = nullptr, t1 = nullptr;
    e = cudaEventCreate(&t0);
    if (e == cudaSuccess) e = cudaEventCreate(&t1);
    if (e == cudaSuccess) e = cudaEventRecord(t0, st);
    for (int r = 0; r < repeat && e == cudaSuccess; ++r) e = conv_launch();
    if (e == cudaSuccess) e = cudaEventRecord(t1, st);
    if (e == cudaSuccess) e = cudaEventSynchronize(t1);
    float ms = 0.f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, t0, t1);
    if (e == cudaSuccess) *ms_out = ms / (float)repeat;
    if (t0) cudaEventDestroy(t0);
    if (t1) cudaEventDestroy(t1);
  }
  if (e == cudaSuccess && mode == 2)
    e = launch_wreduce(reinterpret_cast<const WReduceDesc*>(ws + pl.aux_tab), auxts, n, aux_ts.back(), st);
  if (e == cudaSuccess && !fins.empty())
    e = launch_bn_fin(reinterpret_cast<const BnFinDesc*>(ws + pl.fin_tab), reinterpret_cast<const int*>(ws + pl.fin_ts),
                      (int)fins.size(), fin_ts.back(), st);
  if (e == cudaSuccess && !breds.empty())
    e = launch_bnb_reduce8(reinterpret_cast<const BnBwdDesc*>(ws + pl.red_tab),
                           reinterpret_cast<const int*>(ws + pl.red_ts), (int)breds.size(), red_ts.back(), st);
  if (e == cudaSuccess && !bfins.empty())
    e = launch_bnb_fin(reinterpret_cast<const BnBwdDesc*>(ws + pl.fin_tab), reinterpret_cast<const int*>(ws + pl.fin_ts),
                       (int)bfins.size(), fin_ts.back(), st);
  int32_t host_status = 0;
  if (e == cudaSuccess) e = cudaMemcpyAsync(&host_status, status, sizeof host_status, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return set_last_error(PNN_ECUDA, cudaGetErrorString(e));
  if (host_status == 3) return set_last_error(PNN_ETIMEOUT, "pnn_conv_run: a device wait timed out");
  return PNN_OK;
}
}  // namespace

extern "C" int pnn_conv_run(int32_t mode, int32_t impl, int32_t n, const pnn_conv_args* a, void* workspace,
                            size_t workspace_bytes, void* stream) {
  return conv_run(mode, impl, n, a, workspace, workspace_bytes, stream, 0, nullptr);
}

extern "C" int pnn_conv_time(int32_t mode, int32_t impl, int32_t n, const pnn_conv_args* a, void* workspace,
                             size_t workspace_bytes, void* stream, int32_t repeat, float* ms_per_launch) {
  if (repeat <= 0 || !ms_per_launch) return set_last_error(PNN_EINVAL, "pnn_conv_time: repeat > 0 and an output");
  for (int i = 0; i < n && a; ++i)
    if (a[i].accumulate) return set_last_error(PNN_EINVAL, "pnn_conv_time: accumulating launches are not repeatable");
  return conv_run(mode, impl, n, a, workspace, workspace_bytes, stream, repeat, ms_per_launch);
}
