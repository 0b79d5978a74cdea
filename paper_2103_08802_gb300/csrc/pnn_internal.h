// Internal descriptors shared by the host runtime and the CUDA kernels.
// Every grouped launch receives a device table of per-instance descriptors
// plus a prefix array of tile counts; CTA b belongs to the instance i with
// tile_start[i] <= b < tile_start[i+1].  Tensors are NHWC with the batch
// folded into the row index (row m = (n*H + h)*W + w).
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

namespace pnn {

enum DType : int32_t { DT_F32 = 0, DT_BF16 = 1 };

// A tensor operand.  When scale != nullptr the value read is the "virtual"
// BN(+ReLU) output  v = act(scale[c] * src + shift[c]); zero padding of a
// convolution applies to v, not to src.
struct Src {
  const void* ptr;
  const float* scale;
  const float* shift;
  int32_t dt;
  int32_t relu;
};

struct ConvDesc {
  Src x;                 // forward / wgrad: conv input (maybe virtual)
  const void* w;         // weights [K][R][S][C], dtype w_dt
  int32_t w_dt;
  int32_t B, H, W, C;    // input geometry
  int32_t P, Q, K;       // output geometry
  int32_t R, S, stride, pad;
  // forward epilogue
  void* y; int32_t y_dt;
  const void* res; int32_t res_dt;   // residual added to the output (or null)
  // up to two more addends, out += res2_c[e] * res2[e] (null: none): the
  // parareal correction folded into the conv that produces its operand
  // (r_j = y_j - x_{j+1}, rt_{j+1} = r_{j+1} + F^j(rt_j), ytilde = y_N + rt_N)
  const void* res2[2]; int32_t res2_dt[2]; float res2_c[2];
  float* stats;                       // per-tile BN partials [mtiles][K][2] = (mean, M2) or null
  // dgrad: dx[B*H*W][C] (fp32) = (accumulate ? dx : 0) + W^T * dy
  float* dx; int32_t accumulate;
  // dgrad / wgrad operand dy[B*P*Q][K] (fp32)
  const float* dy;
  // wgrad: partial sums [splits][K][R*S*C]
  float* dw_part;
  int32_t splits, pix_per_split;
  int32_t mtiles, ntiles;             // tile grid of this instance
  int32_t ntile_w;                    // N columns of a tile when ntiles > 1 (256, or 128 TMA-fed)
  int32_t mtile_rows;                 // M rows of a tile: 128, or 256 (TMA-fed weight gradient: two MMA halves)
  int32_t op_bf16;                    // round both contraction operands to bf16 (bf16 mode)
  // TMA-fed tensor-core variant (stride 1): device addresses of two 2-D tensor
  // maps (CUtensorMap, 128-byte aligned) -- tma_a over the A source rows
  // [pixels][channels] (forward: x, dgrad: dy; box min(channels, 64) x 128,
  // no swizzle), tma_b over the bf16 weight rows [N][K] (box 64 x BN,
  // 128-byte swizzle)
  const void* tma_a;
  const void* tma_b;
  // TMA-fed 3x3 forward / data gradient whose tiles lie inside one image
  // (halo_ok): tensor map over the same A source rows with box [halo_rows(W)
  // rows x channels] (no swizzle) -- one box per tile covers all nine taps
  // (null: one box per tap)
  const void* tma_h;
  // TMA-fed forward: tensor map over the output y [pixels][K] (box 16
  // columns x 32 rows, 64-byte swizzle for fp32, 32-byte for bf16), or null
  const void* tma_y;
  // TMA-fed data gradient of a BN(+ReLU) value (x = that virtual value): when
  // bnb_part is set, the epilogue also writes the BN-backward partial sums of
  // its tile, [m-tile][C][2] = (sum g, sum g * xhat) with g = dA masked by the
  // ReLU and xhat = (h - mean) * rstd
  const float* bn_mean;
  const float* bn_rstd;
  float* bnb_part;
};

// out = act( sum_i coef_i * in_i ), optional BN partials of out, NHWC [M][C].
struct EwDesc {
  Src in[3];
  float coef[3];
  int32_t nin;
  void* out; int32_t out_dt;
  int32_t relu;
  float* stats;          // [tiles][C][2] = (mean, M2) or null
  int64_t M;
  int32_t C;
  int32_t rows_per_tile;
  int32_t tiles;
};

// backward of EW: g = dout * [out > 0 if relu]; grad_i (+)= coef_i * g
struct EwBwdDesc {
  const float* dout;
  const void* out; int32_t out_dt; int32_t relu;
  float* gin[3]; float coef[3]; int32_t acc[3];
  int32_t nin;
  int64_t M; int32_t C;
  int32_t rows_per_tile, tiles;
  double* scratch; int32_t* counter; int32_t cgroups, nchunk;  // fin: as for BnFinDesc
};

// BN statistics finalisation: partials[tiles][C][2] -> mean, rstd, scale, shift
constexpr int kFinTilesPerCta = 64;  // BN finalize: partial tiles one CTA adds up (8 per warp)
struct BnFinDesc {
  const float* part;     // [tiles][C][2] = (mean, M2) of each tile's rows
  int32_t tiles, C;
  int64_t count;         // number of rows M
  int32_t rows_per_tile; // rows of every partial tile but the last
  const float* gamma; const float* beta;
  float* mean; float* rstd; float* scale; float* shift;
  float* run_mean; float* run_var;  // running statistics of this BN layer
  float momentum;                   // training: rate at which they follow the batch
  int32_t eval;                     // 1: normalise with the running statistics
  // the reduction over tiles: CTAs = cgroups (32 channels each) x nchunk (64
  // tiles each); chunk sums meet in scratch ([nchunk][C][2] doubles) and the
  // last CTA of a channel group (counter[cg], zero between launches) adds them
  double* scratch; int32_t* counter; int32_t cgroups, nchunk;
};

// BN backward: dz = da * [z > 0 if relu], z = scale*h + shift, xhat = (h-mean)*rstd
//   reduce: part[tile][c] = (sum dz, sum dz*xhat)
//   fin:    dbeta = sum dz, dgamma = sum dz*xhat, coef[c] = (gamma*rstd, dbeta/M, dgamma/M)
//   apply:  dh (+)= gamma*rstd * (dz - dbeta/M - xhat*dgamma/M)
struct BnBwdDesc {
  const float* da;
  const void* h; int32_t h_dt;
  const float* mean; const float* rstd; const float* scale; const float* shift;
  const float* gamma;
  int32_t relu;
  float* part;           // [tiles][C][2]
  float* dgamma; float* dbeta;
  float* coef;           // [C][3]
  float* dh; int32_t accumulate;     // apply: accumulate into dh; fin: into dgamma/dbeta
  const float* add0; const float* add1;  // apply: extra gradients added into dh (residual paths)
  float add_c[2];                          // their coefficients
  int64_t M; int32_t C;
  int32_t rows_per_tile, tiles;
  double* scratch; int32_t* counter; int32_t cgroups, nchunk;  // fin: as for BnFinDesc
};

struct PoolDesc {
  Src x;                 // input (maybe virtual)
  void* y; int32_t y_dt; // output
  int32_t B, H, W, C, P, Q, k, stride, pad;
  // backward: dx (+)= route(dy)
  const float* dy; float* dx; int32_t accumulate;
  int32_t tiles;
};

// wgrad split reduction: dw[K*RSC] = sum_s part[s][K*RSC]
// wgrad split reduction: dw[K*RSC] = sum_s part[s][...]; partials are laid out
// [s][K][RSC] (CUDA-core wgrad) or [s][RSC][K] (tensor-core wgrad, transposed = 1)
struct WReduceDesc {
  const float* part;
  float* dw;
  int32_t splits;
  int32_t accumulate;
  int64_t n;
  int32_t tiles;
  int32_t transposed, kout, rsc;
};

// bf16 weight transpose for the tensor-core data gradient: dst[c][r][s][k] = src[k][r][s][c]
struct WtDesc {
  const void* src;
  void* dst;
  int32_t K, RS, C;
  int64_t n;
};

// generic strided fp32 GEMM: C[m][n] = beta*C + sum_k A[m*sam + k*sak] * B[k*sbk + n*sbn] (+ bias[n]) (relu)
struct GemmDesc {
  const float* A; const float* Bm; float* Cm;
  const float* bias;
  int32_t M, N, K;
  int64_t sam, sak, sbk, sbn, scm;
  float beta;
  int32_t relu;
  int32_t mtiles, ntiles;
};

// ------------------------------------------------------------ launchers
// All launchers enqueue on `st` and return cudaGetLastError().
cudaError_t launch_conv_fwd_simt(const ConvDesc* tab, const int* tstart, int n, int total_tiles,
                                 int variant, cudaStream_t st);
cudaError_t launch_conv_dgrad_simt(const ConvDesc* tab, const int* tstart, int n, int total_tiles,
                                   int variant, cudaStream_t st);
// variant 1: few input channels (R*S*C <= 64), im2col staged per 64-pixel step
cudaError_t launch_conv_wgrad_simt(const ConvDesc* tab, const int* tstart, int n, int total_tiles, int variant,
                                   cudaStream_t st);
cudaError_t launch_wreduce(const WReduceDesc* tab, const int* tstart, int n, int total_tiles, cudaStream_t st);
cudaError_t launch_ew(const EwDesc* tab, const int* tstart, int n, int total_tiles, cudaStream_t st);
cudaError_t launch_ew_bwd(const EwBwdDesc* tab, const int* tstart, int n, int total_tiles, cudaStream_t st);
cudaError_t launch_bn_fin(const BnFinDesc* tab, const int* tstart, int n, int total_tiles, cudaStream_t st);
cudaError_t launch_bnb_reduce(const BnBwdDesc* tab, const int* tstart, int n, int total_tiles, cudaStream_t st);
cudaError_t launch_bnb_fin(const BnBwdDesc* tab, const int* tstart, int n, int total_tiles, cudaStream_t st);
cudaError_t launch_bnb_apply(const BnBwdDesc* tab, const int* tstart, int n, int total_tiles, cudaStream_t st);
// 8 channels per thread; every instance needs C % 8 == 0 and C <= 2048
cudaError_t launch_bnb_reduce8(const BnBwdDesc* tab, const int* tstart, int n, int total_tiles, cudaStream_t st);
cudaError_t launch_bnb_apply8(const BnBwdDesc* tab, const int* tstart, int n, int total_tiles, cudaStream_t st);
cudaError_t launch_pool_fwd(const PoolDesc* tab, const int* tstart, int n, int total_tiles, cudaStream_t st);
cudaError_t launch_pool_bwd(const PoolDesc* tab, const int* tstart, int n, int total_tiles, cudaStream_t st);
cudaError_t launch_gemm(const GemmDesc* tab, const int* tstart, int n, int total_tiles, cudaStream_t st);
// tcgen05 implicit-GEMM convolution (bf16 operands, fp32 accumulate in TMEM);
// instances need C % 8 == 0; bnmax = largest N tile (multiple of 16, <= 256)
// (max_ctas > 0 caps the persistent grid below the SM count, leaving SMs to
// launches of other streams)
cudaError_t launch_conv_fwd_tc(const ConvDesc* tab, const int* tstart, int n, int total_tiles, int bnmax,
                               int32_t* status, cudaStream_t st, int max_ctas = 0);
cudaError_t launch_conv_dgrad_tc(const ConvDesc* tab, const int* tstart, int n, int total_tiles, int bnmax,
                                 int32_t* status, cudaStream_t st, int max_ctas = 0);
cudaError_t launch_conv_wgrad_tc(const ConvDesc* tab, const int* tstart, int n, int total_tiles, int bnmax,
                                 int32_t* status, cudaStream_t st, int max_ctas = 0);
// TMA-fed stride-1 forward (mode 0), data-gradient (mode 1) or weight-gradient
// (mode 2) tensor-core conv; raw_bytes: one pipeline stage's raw slot (the
// largest over the launch's instances, a multiple of 1024); op_bytes: one
// stage's operand slot when the launch has halo tiles (the larger of
// halo_op_bytes and the default slot), 0 for the default slot
// wide: every tile of the launch is one k-step (the epilogue bounds the
// kernel): the variant with three epilogue groups and two transform warps
cudaError_t launch_conv_tma(int mode, int wide, const ConvDesc* tab, const int* tstart, int n, int total, int bnmax,
                            int raw_bytes, int op_bytes, int32_t* status, cudaStream_t st, int max_ctas = 0);
// whether the TMA-fed kernel of `mode` holds at least two stages of this size
bool conv_tma_fits(int mode, int bnmax, int raw_bytes, int op_bytes = 0);
// the default operand slot of a TMA-fed stage (A then bnmax weight rows)
int conv_tma_op_bytes(int mode, int bnmax);
// whether a halo instance (mode 0 or 1; A source W x ch, N tile bn) leaves
// two stages even beside per-tap instances of the same launch
bool conv_halo_fits(int mode, int W, int ch, int bn);
// record a message for pnn_last_error(NULL) and return `code`
int set_last_error(int code, const char* msg);
// streaming multiprocessors of the current device, queried once per device
// (thread-safe); 1 if the query fails, which keeps every grid valid
int device_sm_count();
// cudaFuncSetAttribute(MaxDynamicSharedMemorySize) once per (device, kernel
// slot < 32); thread-safe
cudaError_t set_smem_attr_once(int slot, const void* kernel, int bytes);

// debug builds: first misaligned vector access of the tensor-core kernels (0 = none)
unsigned long long conv_tc_debug_word();
cudaError_t launch_wtrans(const WtDesc* tab, const int* tstart, int n, int total_tiles, cudaStream_t st);
constexpr int kTcBM = 128;

// single-instance helpers
cudaError_t launch_pack_input(const float* x_nchw, void* out, int32_t out_dt, int B, int C, int H, int W,
                              cudaStream_t st);
cudaError_t launch_gap(Src x, float* feat, int B, int HW, int C, cudaStream_t st);
cudaError_t launch_gap_bwd(const float* dfeat, float* dx, int B, int HW, int C, cudaStream_t st);
cudaError_t launch_softmax_ce(const float* logits, const int32_t* labels, int B, int m, float* loss,
                              float* dlogits, int32_t* status, cudaStream_t st);
cudaError_t launch_colsum(const float* A, int rows, int cols, float* out, cudaStream_t st);
cudaError_t launch_relu_mask(float* g, const float* pre, int64_t n, cudaStream_t st);
cudaError_t launch_sgd(float* w, const float* g, float* v, void* shadow, int32_t shadow_dt, int64_t n,
                       float lr, float mu, float wd, int nesterov, int first, cudaStream_t st);
cudaError_t launch_export(Src x, int B, int H, int W, int C, float* out_nchw, cudaStream_t st);
cudaError_t launch_copy_cast(const float* in, void* out, int32_t out_dt, int64_t n, cudaStream_t st);
cudaError_t launch_weight_cast(const float* in, void* out, int32_t out_dt, int64_t n, cudaStream_t st);

// tile geometry helpers shared by runtime and kernels
constexpr int kEwRowsPerTile = 64;
#ifdef __CUDACC__
#define PNN_HD __host__ __device__
#else
#define PNN_HD
#endif
// BN forward statistics are kept as (count, mean, M2 = sum of squared
// deviations from the mean) and combined with the pairwise update of Chan,
// Golub & LeVeque ("Updating formulae and a pairwise algorithm for computing
// sample variances", 1979): for disjoint sets a and b with n = n_a + n_b and
// delta = mean_b - mean_a,
//   mean = mean_a + delta * n_b / n,   M2 = M2_a + M2_b + delta^2 * n_a * n_b / n,
// which never subtracts two large sums (the one-pass sum(h^2) - n * mean^2
// loses the variance when |mean| >> std).  Per-tile partials are
// [tiles][C][2] = (mean, M2) of the tile's rows; a tile's count follows from
// its row range.
template <typename T>
PNN_HD inline void chan_merge(T& n, T& mean, T& m2, T nb, T meanb, T m2b) {
  if (nb <= T(0)) return;
  if (n <= T(0)) { n = nb; mean = meanb; m2 = m2b; return; }
  const T nn = n + nb;
  const T delta = meanb - mean;
  const T f = nb / nn;
  mean = mean + delta * f;
  m2 = m2 + m2b + delta * delta * n * f;
  n = nn;
}

// TMA-fed weight gradient: the two boxes of a k-step (64 pixels) -- the
// activation rows of every tap (halo of pad*W + pad rows each side) x cwx
// channels, and the output-gradient rows x K -- and their raw-slot offsets
struct WgBoxes {
  int halo, hrows, cwx, escx, xbytes, yoff, ybytes;
};
PNN_HD inline WgBoxes wg_boxes(int C, int K, int W, int pad, bool xbf) {
  WgBoxes b;
  b.halo = pad * W + pad;
  b.hrows = 64 + 2 * b.halo;
  b.cwx = C <= 64 ? C : 128;
  b.escx = xbf ? 2 : 4;
  b.xbytes = b.hrows * b.cwx * b.escx;
  b.yoff = (b.xbytes + 127) & ~127;
  b.ybytes = 64 * K * 4;
  return b;
}
PNN_HD inline int wg_raw_bytes(const WgBoxes& b) { return (b.yoff + b.ybytes + 1023) & ~1023; }

// TMA-fed 3x3 forward / data gradient, halo tiles.  A 128-pixel tile that
// lies inside one image reads input pixels m0 - W - 1 .. m0 + 128 + W: one
// box of halo_rows(W) rows.  The transform forms three copies of it, one per
// column offset s' in {-1, 0, 1}, each of 128 + 2W rows (copy s' row j =
// pixel m0 - W + s' + j, zero where that pixel lies outside the tile's image
// or where the output column x - s' would leave the row), in the
// no-swizzle K-major layout: one plane of 16-byte rows per 8 channels.  Tap
// (r', s') is then copy s' from row (r' + 1) W: a descriptor offset, for any
// W.  Needs 128 | H*W (no tile crosses an image), W <= 63 (a TMA box holds
// at most 256 rows) and 16 | channels <= 64.
PNN_HD inline bool halo_ok(int k, int stride, int pad, int H, int W, int ch) {
  return k == 3 && stride == 1 && pad == 1 && W > 0 && (H * W) % kTcBM == 0 && kTcBM + 2 * W + 2 <= 256 &&
         ch % 16 == 0 && ch <= 64;
}
PNN_HD inline int halo_rows(int W) { return kTcBM + 2 * W + 2; }
PNN_HD inline int halo_plane_bytes(int W) { return (kTcBM + 2 * W) * 16; }
PNN_HD inline int halo_copy_bytes(int W, int ch) { return (ch / 8) * halo_plane_bytes(W); }
// weight boxes of a halo tile: the tile's whole K = 9 * ch in boxes of 64
PNN_HD inline int halo_nbox(int ch) { return (9 * ch + 63) / 64; }
PNN_HD inline int halo_raw_bytes(int W, int ch, int esz) { return (halo_rows(W) * ch * esz + 1023) & ~1023; }
// operand slot of a halo tile: the weight boxes (bn rows each), then the three copies
PNN_HD inline int halo_op_bytes(int W, int ch, int bn) {
  return (halo_nbox(ch) * bn * 128 + 3 * halo_copy_bytes(W, ch) + 1023) & ~1023;
}

// ---------------------------------------------------------------- conv kernel choice
// (mode 0 forward, 1 data gradient, 2 weight gradient; variant 1 = TMA-fed,
// 0 = thread-gathered tensor-core kernel)
// The TMA-fed forward / data gradient load each filter tap as one
// [128 rows x min(channels, 64)] box: stride 1, same padding, and a channel
// count (of the A source) that divides 64 or is a multiple of it.
inline bool tma_shape_ok(int k, int stride, int pad, int ch) {
  const bool geom = stride == 1 && ((k == 1 && pad == 0) || (k == 3 && pad == 1));
  return geom && ch % 8 == 0 && (ch <= 64 ? 64 % ch == 0 : ch % 64 == 0);
}
// N columns of a tile when the layer needs several: 128 for the TMA-fed
// forward and data gradient (a smaller operand slot leaves room for more
// pipeline stages), 256 otherwise.
inline int tc_ntile_cols(int mode, int variant) { return variant == 1 && mode != 2 ? 128 : 256; }
// M rows of a tile: 256 for the TMA-fed weight gradient of a layer with at
// most 128 input channels (two MMA halves share each B operand, so a layer
// with up to 256 (r,s,c) rows makes one pass over the pixels; a tile then
// holds whole taps, all inside the activation box), 128 otherwise.
inline int tc_tile_rows(int mode, int variant, int C) { return mode == 2 && variant == 1 && C <= 128 ? 256 : kTcBM; }
// 2-D tensor map (CUtensorMap, 128 bytes at `map`) over rows x inner elements
// (bf16 or fp32, row pitch inner * element size) with box
// [box_rows][box_inner]; swz: swizzle span in bytes (128, 64, 32 or 0).
// Returns 0, or non-zero with a message in *why.
int encode_tensor_map_2d(void* map, const void* base, bool bf16, int64_t inner, int64_t rows, int box_inner,
                         int box_rows, int swz, const char** why);

constexpr int kBnbRowsPerTile = 256;  // BN backward reduce/apply tiles: at least this many rows
// rows of a BN-backward tile for C channels: about 32K elements a CTA
inline int bnb_rows_per_tile(int C) { return C > 0 && 32768 / C > kBnbRowsPerTile ? 32768 / C : kBnbRowsPerTile; }
// The TMA-fed weight gradient loads a k-step's activation rows for all taps
// as one halo box and the output-gradient rows as another: channels 8..64
// (dividing 64) or multiples of 128 up to 512, at most 128 output channels
// (one N tile), a halo of at most 256 rows, and two stages in shared memory.
inline bool tma_wgrad_ok(int k, int stride, int pad, int C, int K, int W, bool xbf) {
  if (!(stride == 1 && ((k == 1 && pad == 0) || (k == 3 && pad == 1)))) return false;
  if (!(C % 8 == 0 && ((C <= 64 && 64 % C == 0) || (C % 128 == 0 && C <= 512)))) return false;
  if (K % 8 != 0 || K > 128) return false;
  const WgBoxes b = wg_boxes(C, K, W, pad, xbf);
  return b.hrows <= 256 && conv_tma_fits(2, 128, wg_raw_bytes(b));
}
struct ConvTile { int BM, BN; };
inline ConvTile simt_tile(int variant) {
  return variant == 0 ? ConvTile{64, 64} : (variant == 1 ? ConvTile{128, 32} : ConvTile{256, 16});
}
constexpr int kWgradBM = 64, kWgradBN = 64, kWgradBK = 16;

}  // namespace pnn
