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
  float* stats;                       // per-tile BN partials [mtiles][K][2] or null
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
  float* stats;          // [tiles][C][2] or null
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
  const float* part;
  int32_t tiles, C;
  int64_t count;         // number of rows M
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
cudaError_t launch_conv_wgrad_simt(const ConvDesc* tab, const int* tstart, int n, int total_tiles,
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
// largest over the launch's instances, a multiple of 1024)
cudaError_t launch_conv_tma(int mode, const ConvDesc* tab, const int* tstart, int n, int total, int bnmax,
                            int raw_bytes, int32_t* status, cudaStream_t st, int max_ctas = 0);
// whether the TMA-fed kernel of `mode` holds at least two stages of this size
bool conv_tma_fits(int mode, int bnmax, int raw_bytes);
// record a message for pnn_last_error(NULL) and return `code`
int set_last_error(int code, const char* msg);

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

constexpr int kBnbRowsPerTile = 256;  // BN backward reduce/apply tiles: at least this many rows
// rows of a BN-backward tile for C channels: about 32K elements a CTA
inline int bnb_rows_per_tile(int C) { return C > 0 && 32768 / C > kBnbRowsPerTile ? 32768 / C : kBnbRowsPerTile; }
struct ConvTile { int BM, BN; };
inline ConvTile simt_tile(int variant) {
  return variant == 0 ? ConvTile{64, 64} : (variant == 1 ? ConvTile{128, 32} : ConvTile{256, 16});
}
constexpr int kWgradBM = 64, kWgradBN = 64, kWgradBK = 16;

}  // namespace pnn
