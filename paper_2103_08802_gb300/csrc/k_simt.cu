// CUDA-core kernels of the parareal training step: implicit-GEMM convolution
// (forward, data gradient, weight gradient) used in fp32 check mode, and every
// non-convolution op of the step (BN statistics and backward, elementwise
// correction/residual ops, pooling, head, loss, SGD) used in both precisions.
//
// Every kernel is "grouped": one launch covers a list of independent problem
// instances (typically the same layer position of all N fine subnetworks,
// Algorithm 1's parallel loop), each CTA finds its instance from a tile prefix.
// All reductions run in a fixed order so that results are bit-reproducible.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <mutex>

#include "pnn_internal.h"

namespace pnn {

// ---------------------------------------------------------------- helpers
__device__ __forceinline__ float ldv(const void* p, int dt, int64_t i) {
  return dt == DT_F32 ? __ldg(reinterpret_cast<const float*>(p) + i)
                      : __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(p)[i]);
}
__device__ __forceinline__ float rnd(int dt, float v) {
  return dt == DT_BF16 ? __bfloat162float(__float2bfloat16_rn(v)) : v;
}
__device__ __forceinline__ void stv(void* p, int dt, int64_t i, float v) {
  if (dt == DT_F32) reinterpret_cast<float*>(p)[i] = v;
  else reinterpret_cast<__nv_bfloat16*>(p)[i] = __float2bfloat16_rn(v);
}
__device__ __forceinline__ float ld_src(const Src& s, int64_t i, int c) {
  float v = ldv(s.ptr, s.dt, i);
  if (s.scale) {
    v = fmaf(__ldg(s.scale + c), v, __ldg(s.shift + c));
    if (s.relu) v = fmaxf(v, 0.f);
  }
  return v;
}
// index of the instance that owns CTA b: the largest i with tstart[i] <= b
// (every thread of the block calls it with the same b: up to 32 instances
// the warp reads the starts at once and counts those <= b -- one dependent
// load instead of log2(n) -- else a binary search)
__device__ __forceinline__ int find_instance(const int* tstart, int n, int b) {
  if (n <= 32) {
    const int lane = threadIdx.x & 31;
    const bool le = lane < n && __ldg(tstart + lane) <= b;
    return __popc(__ballot_sync(0xffffffffu, le)) - 1;
  }
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (__ldg(tstart + mid) <= b) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// ---------------------------------------------------------------- conv fwd
// Y[m][k] = sum_{r,s,c} act(X)[n, p*st+r-pad, q*st+s-pad, c] * W[k][r][s][c] (+ res[m][k])
template <int BM, int BN>
__global__ void __launch_bounds__(256) k_conv_fwd(const ConvDesc* __restrict__ tab,
                                                  const int* __restrict__ tstart, int n) {
  constexpr int BK = 16, TM = BM / 16, TN = BN / 16;
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  __shared__ float red[16][BN][2];
  const int inst = find_instance(tstart, n, blockIdx.x);
  const ConvDesc& d = tab[inst];
  const int t = blockIdx.x - tstart[inst];
  const int tm = t % d.mtiles, tn = t / d.mtiles;
  const int M = d.B * d.P * d.Q, Kt = d.R * d.S * d.C;
  const int m0 = tm * BM, n0 = tn * BN;
  const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
  float acc[TM][TN];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;

  for (int k0 = 0; k0 < Kt; k0 += BK) {
    for (int e = tid; e < BM * BK; e += 256) {
      const int kk = e % BK, mm = e / BK;
      const int m = m0 + mm, k = k0 + kk;
      float v = 0.f;
      if (m < M && k < Kt) {
        const int c = k % d.C, rs = k / d.C, s = rs % d.S, r = rs / d.S;
        const int q = m % d.Q, tmp = m / d.Q, p = tmp % d.P, nb = tmp / d.P;
        const int h = p * d.stride + r - d.pad, w = q * d.stride + s - d.pad;
        if (h >= 0 && h < d.H && w >= 0 && w < d.W)
          v = ld_src(d.x, ((int64_t)(nb * d.H + h) * d.W + w) * d.C + c, c);
      }
      As[kk][mm] = d.op_bf16 ? rnd(DT_BF16, v) : v;
    }
    for (int e = tid; e < BN * BK; e += 256) {
      const int kk = e % BK, nn = e / BK;
      const int k = k0 + kk, co = n0 + nn;
      Bs[kk][nn] = (k < Kt && co < d.K) ? ldv(d.w, d.w_dt, (int64_t)co * Kt + k) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      float a[TM], b[TN];
#pragma unroll
      for (int i = 0; i < TM; ++i) a[i] = As[kk][ty + 16 * i];
#pragma unroll
      for (int j = 0; j < TN; ++j) b[j] = Bs[kk][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  // epilogue: residual, store, BN partials (mean, M2) of the stored value:
  // two passes over each thread's TM rows, then chan_merge over the 16 row
  // groups in order
  int cnt = 0;  // rows of this thread inside the layer
#pragma unroll
  for (int i = 0; i < TM; ++i) cnt += m0 + ty + 16 * i < M ? 1 : 0;
#pragma unroll
  for (int j = 0; j < TN; ++j) {
    const int co = n0 + tx + 16 * j;
    float s1 = 0.f;
#pragma unroll
    for (int i = 0; i < TM; ++i) {
      const int m = m0 + ty + 16 * i;
      if (m < M && co < d.K) {
        const int64_t o = (int64_t)m * d.K + co;
        float v = acc[i][j];
        if (d.res) v += ldv(d.res, d.res_dt, o);
        if (d.res2[0]) v = fmaf(d.res2_c[0], ldv(d.res2[0], d.res2_dt[0], o), v);
        if (d.res2[1]) v = fmaf(d.res2_c[1], ldv(d.res2[1], d.res2_dt[1], o), v);
        v = rnd(d.y_dt, v);
        stv(d.y, d.y_dt, o, v);
        acc[i][j] = v;
        s1 += v;
      }
    }
    const float mean = cnt > 0 ? s1 / (float)cnt : 0.f;
    float m2 = 0.f;
#pragma unroll
    for (int i = 0; i < TM; ++i)
      if (m0 + ty + 16 * i < M) m2 = fmaf(acc[i][j] - mean, acc[i][j] - mean, m2);
    red[ty][tx + 16 * j][0] = mean;
    red[ty][tx + 16 * j][1] = m2;
  }
  if (d.stats) {
    __syncthreads();
    for (int nn = tid; nn < BN; nn += 256) {
      const int co = n0 + nn;
      if (co < d.K) {
        float n = 0.f, mean = 0.f, m2 = 0.f;
        for (int r = 0; r < 16; ++r) {
          int cr = 0;
          for (int i = 0; i < TM; ++i) cr += m0 + r + 16 * i < M ? 1 : 0;
          chan_merge(n, mean, m2, (float)cr, red[r][nn][0], red[r][nn][1]);
        }
        d.stats[((int64_t)tm * d.K + co) * 2 + 0] = mean;
        d.stats[((int64_t)tm * d.K + co) * 2 + 1] = m2;
      }
    }
  }
}

// ---------------------------------------------------------------- conv dgrad
// dX[m=(n,h,w)][c] (+)= sum_{r,s,k} dY[n, (h+pad-r)/st, (w+pad-s)/st, k] * W[k][r][s][c]
// (terms whose division is inexact or out of range are zero)
template <int BM, int BN>
__global__ void __launch_bounds__(256) k_conv_dgrad(const ConvDesc* __restrict__ tab,
                                                    const int* __restrict__ tstart, int n) {
  constexpr int BK = 16, TM = BM / 16, TN = BN / 16;
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int inst = find_instance(tstart, n, blockIdx.x);
  const ConvDesc& d = tab[inst];
  const int t = blockIdx.x - tstart[inst];
  const int tm = t % d.mtiles, tn = t / d.mtiles;
  const int M = d.B * d.H * d.W, Kt = d.R * d.S * d.K;
  const int m0 = tm * BM, n0 = tn * BN;
  const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
  float acc[TM][TN];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < Kt; k0 += BK) {
    for (int e = tid; e < BM * BK; e += 256) {
      const int kk = e % BK, mm = e / BK;
      const int m = m0 + mm, k = k0 + kk;
      float v = 0.f;
      if (m < M && k < Kt) {
        const int ko = k % d.K, rs = k / d.K, s = rs % d.S, r = rs / d.S;
        const int w = m % d.W, tmp = m / d.W, h = tmp % d.H, nb = tmp / d.H;
        const int pn = h + d.pad - r, qn = w + d.pad - s;
        if (pn >= 0 && qn >= 0 && pn % d.stride == 0 && qn % d.stride == 0) {
          const int p = pn / d.stride, q = qn / d.stride;
          if (p < d.P && q < d.Q) v = __ldg(d.dy + ((int64_t)(nb * d.P + p) * d.Q + q) * d.K + ko);
        }
      }
      As[kk][mm] = d.op_bf16 ? rnd(DT_BF16, v) : v;
    }
    for (int e = tid; e < BN * BK; e += 256) {
      const int nn = e % BN, kk = e / BN;
      const int k = k0 + kk, c = n0 + nn;
      float v = 0.f;
      if (k < Kt && c < d.C) {
        const int ko = k % d.K, rs = k / d.K;
        v = ldv(d.w, d.w_dt, ((int64_t)ko * d.R * d.S + rs) * d.C + c);
      }
      Bs[kk][nn] = v;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      float a[TM], b[TN];
#pragma unroll
      for (int i = 0; i < TM; ++i) a[i] = As[kk][ty + 16 * i];
#pragma unroll
      for (int j = 0; j < TN; ++j) b[j] = Bs[kk][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < TM; ++i) {
    const int m = m0 + ty + 16 * i;
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int c = n0 + tx + 16 * j;
      if (m < M && c < d.C) {
        const int64_t o = (int64_t)m * d.C + c;
        d.dx[o] = d.accumulate ? d.dx[o] + acc[i][j] : acc[i][j];
      }
    }
  }
}

// ---------------------------------------------------------------- conv wgrad
// part[split][k][(r,s,c)] = sum_{m in split} dY[m][k] * act(X)[n, p*st+r-pad, q*st+s-pad, c]
__global__ void __launch_bounds__(256) k_conv_wgrad(const ConvDesc* __restrict__ tab,
                                                    const int* __restrict__ tstart, int n) {
  constexpr int BM = kWgradBM, BN = kWgradBN, BK = kWgradBK, TM = BM / 16, TN = BN / 16;
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int inst = find_instance(tstart, n, blockIdx.x);
  const ConvDesc& d = tab[inst];
  int t = blockIdx.x - tstart[inst];
  const int tm = t % d.mtiles;
  t /= d.mtiles;
  const int tn = t % d.ntiles, split = t / d.ntiles;
  const int RSC = d.R * d.S * d.C, Mp = d.B * d.P * d.Q;
  const int m0 = tm * BM, n0 = tn * BN;
  const int p_begin = split * d.pix_per_split;
  const int p_end = min(Mp, p_begin + d.pix_per_split);
  const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
  float acc[TM][TN];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;
  for (int k0 = p_begin; k0 < p_end; k0 += BK) {
    for (int e = tid; e < BM * BK; e += 256) {
      const int mm = e % BM, kk = e / BM;
      const int ko = m0 + mm, pix = k0 + kk;
      const float v = (ko < d.K && pix < p_end) ? __ldg(d.dy + (int64_t)pix * d.K + ko) : 0.f;
      As[kk][mm] = d.op_bf16 ? rnd(DT_BF16, v) : v;
    }
    for (int e = tid; e < BN * BK; e += 256) {
      const int nn = e % BN, kk = e / BN;
      const int j = n0 + nn, pix = k0 + kk;
      float v = 0.f;
      if (j < RSC && pix < p_end) {
        const int c = j % d.C, rs = j / d.C, s = rs % d.S, r = rs / d.S;
        const int q = pix % d.Q, tmp = pix / d.Q, p = tmp % d.P, nb = tmp / d.P;
        const int h = p * d.stride + r - d.pad, w = q * d.stride + s - d.pad;
        if (h >= 0 && h < d.H && w >= 0 && w < d.W)
          v = ld_src(d.x, ((int64_t)(nb * d.H + h) * d.W + w) * d.C + c, c);
      }
      Bs[kk][nn] = d.op_bf16 ? rnd(DT_BF16, v) : v;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      float a[TM], b[TN];
#pragma unroll
      for (int i = 0; i < TM; ++i) a[i] = As[kk][ty + 16 * i];
#pragma unroll
      for (int j = 0; j < TN; ++j) b[j] = Bs[kk][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  float* out = d.dw_part + (int64_t)split * d.K * RSC;
#pragma unroll
  for (int i = 0; i < TM; ++i) {
    const int ko = m0 + ty + 16 * i;
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int jj = n0 + tx + 16 * j;
      if (ko < d.K && jj < RSC) out[(int64_t)ko * RSC + jj] = acc[i][j];
    }
  }
}

// Weight gradient of a conv with few input channels (the 3-channel stem and
// C^j convs, R*S*C <= 64): the same tiles, splits and partial layout as
// k_conv_wgrad, but each 64-pixel step stages dY [64 px][64 k_out] and the
// im2col operand [64 px][R*S*C] once in shared memory (pixel and (r,s,c)
// coordinates from per-CTA tables instead of divisions per element), and
// thread t accumulates outputs (k, j) = t, t + 256, ... of the tile over the
// step's pixels in order.
__global__ void __launch_bounds__(256) k_conv_wgrad_small(const ConvDesc* __restrict__ tab,
                                                          const int* __restrict__ tstart, int n) {
  constexpr int BM = kWgradBM, BN = kWgradBN, BP = 64, MAXO = (BM * BN) / 256;
  __shared__ float As[BP][BM + 1];  // dY[pixel][k_out]
  __shared__ float Bs[BP][BN + 1];  // im2col[pixel][j]
  __shared__ int jr[BN], js[BN], jc[BN];
  __shared__ int pn[BP], ph[BP], pw[BP];
  const int inst = find_instance(tstart, n, blockIdx.x);
  const ConvDesc& d = tab[inst];
  int t = blockIdx.x - tstart[inst];
  const int tm = t % d.mtiles;
  t /= d.mtiles;
  const int tn = t % d.ntiles, split = t / d.ntiles;
  const int RSC = d.R * d.S * d.C, Mp = d.B * d.P * d.Q;
  const int m0 = tm * BM, n0 = tn * BN;
  const int km = min(BM, d.K - m0), jn = min(BN, RSC - n0);
  const int p_begin = split * d.pix_per_split;
  const int p_end = min(Mp, p_begin + d.pix_per_split);
  const int tid = threadIdx.x;
  for (int j = tid; j < jn; j += 256) {
    const int jj = n0 + j, c = jj % d.C, rs = jj / d.C;
    jr[j] = rs / d.S - d.pad;
    js[j] = rs % d.S - d.pad;
    jc[j] = c;
  }
  float acc[MAXO];
#pragma unroll
  for (int i = 0; i < MAXO; ++i) acc[i] = 0.f;
  for (int k0 = p_begin; k0 < p_end; k0 += BP) {
    __syncthreads();  // the previous step's tiles are consumed
    if (tid < BP) {
      const int pix = k0 + tid;
      const int q = pix % d.Q, tmp = pix / d.Q, pp = tmp % d.P;
      pn[tid] = pix < p_end ? tmp / d.P : -1;
      ph[tid] = pp * d.stride;
      pw[tid] = q * d.stride;
    }
    __syncthreads();
    for (int e = tid; e < BP * BM; e += 256) {
      const int kk = e % BM, px = e / BM;
      const float v = (kk < km && pn[px] >= 0) ? __ldg(d.dy + (int64_t)(k0 + px) * d.K + m0 + kk) : 0.f;
      As[px][kk] = d.op_bf16 ? rnd(DT_BF16, v) : v;
    }
    for (int e = tid; e < BP * BN; e += 256) {
      const int j = e % BN, px = e / BN;
      float v = 0.f;
      if (j < jn && pn[px] >= 0) {
        const int h = ph[px] + jr[j], w = pw[px] + js[j];
        if (h >= 0 && h < d.H && w >= 0 && w < d.W)
          v = ld_src(d.x, ((int64_t)(pn[px] * d.H + h) * d.W + w) * d.C + jc[j], jc[j]);
      }
      Bs[px][j] = d.op_bf16 ? rnd(DT_BF16, v) : v;
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < MAXO; ++i) {
      const int o = tid + 256 * i;
      if (o >= km * jn) break;
      const int k = o / jn, j = o - k * jn;
      float a = acc[i];
      for (int px = 0; px < BP; ++px) a = fmaf(As[px][k], Bs[px][j], a);
      acc[i] = a;
    }
  }
  float* out = d.dw_part + (int64_t)split * d.K * RSC;
#pragma unroll
  for (int i = 0; i < MAXO; ++i) {
    const int o = tid + 256 * i;
    if (o >= km * jn) break;
    const int k = o / jn, j = o - k * jn;
    out[(int64_t)(m0 + k) * RSC + n0 + j] = acc[i];
  }
}

// 32 elements per CTA, 8 lanes per element: lane l sums splits l, l+8, ...
// in order, then a fixed xor-shuffle tree combines the 8 lanes.
// 32 consecutive partial positions e per CTA; warp w sums splits w, w+8, ..
// (coalesced 128-byte rows of one split), then the eight warp sums are added
// in warp order: a fixed order, so the result is deterministic.  Transposed
// partials ([split][j][k_out], the tensor-core layout) land in dw[k_out][j].
__global__ void __launch_bounds__(256) k_wreduce(const WReduceDesc* __restrict__ tab, const int* __restrict__ tstart,
                                                 int n) {
  __shared__ float red[8][32];
  const int inst = find_instance(tstart, n, blockIdx.x);
  const WReduceDesc d = tab[inst];
  const int64_t e = (int64_t)(blockIdx.x - tstart[inst]) * 32 + (threadIdx.x & 31);
  const int w = threadIdx.x >> 5;
  float s = 0.f;
  if (e < d.n)
    for (int k = w; k < d.splits; k += 8) s += d.part[(int64_t)k * d.n + e];
  red[w][threadIdx.x & 31] = s;
  __syncthreads();
  if (w == 0 && e < d.n) {
    float t = red[0][threadIdx.x];
#pragma unroll
    for (int i = 1; i < 8; ++i) t += red[i][threadIdx.x];
    const int64_t i = d.transposed ? (e % d.kout) * d.rsc + e / d.kout : e;
    d.dw[i] = d.accumulate ? d.dw[i] + t : t;
  }
}

__global__ void k_wtrans(const WtDesc* __restrict__ tab, const int* __restrict__ tstart, int n) {
  const int inst = find_instance(tstart, n, blockIdx.x);
  const WtDesc& d = tab[inst];
  const int64_t i = (int64_t)(blockIdx.x - tstart[inst]) * blockDim.x + threadIdx.x;
  if (i >= d.n) return;
  const int k = (int)(i % d.K);
  const int64_t t = i / d.K;
  const int rs = (int)(t % d.RS);
  const int c = (int)(t / d.RS);
  reinterpret_cast<__nv_bfloat16*>(d.dst)[i] =
      reinterpret_cast<const __nv_bfloat16*>(d.src)[((int64_t)k * d.RS + rs) * d.C + c];
}

// ---------------------------------------------------------------- row-tile geometry
// A tile is rows_per_tile rows x all C channels.  For C <= 256 (a power of
// two) thread t owns channel t % C and rows t / C + g * (256 / C); for
// C > 256 it owns channels t + 256 i and all rows.
struct RowTile {
  int G, cpt, c0, g;
  __device__ RowTile(int C, int tid) {
    if (C <= 256) {
      G = 256 / C; cpt = 1; c0 = tid % C; g = tid / C;
      if (g >= G) c0 = C;  // idle thread (C does not divide 256)
    } else { G = 1; cpt = (C + 255) / 256; c0 = tid; g = 0; }
  }
};

__global__ void __launch_bounds__(256) k_ew(const EwDesc* __restrict__ tab, const int* __restrict__ tstart, int n) {
  __shared__ float red[256][2];
  const int inst = find_instance(tstart, n, blockIdx.x);
  const EwDesc& d = tab[inst];
  const int tile = blockIdx.x - tstart[inst];
  const int C = d.C;
  const RowTile rt(C, threadIdx.x);
  const int64_t r0 = (int64_t)tile * d.rows_per_tile;
  const int64_t r1 = min((int64_t)d.M, r0 + d.rows_per_tile);
  // BN partials of the output: Welford's update over this thread's rows
  // (count, mean, M2), then chan_merge over the row groups in order
  for (int ci = 0; ci < rt.cpt; ++ci) {
    const int c = rt.c0 + 256 * ci;
    float n = 0.f, mean = 0.f, m2 = 0.f;
    if (c < C) {
      for (int64_t r = r0 + rt.g; r < r1; r += rt.G) {
        const int64_t o = r * C + c;
        float v = 0.f;
        for (int i = 0; i < d.nin; ++i) v = fmaf(d.coef[i], ld_src(d.in[i], o, c), v);
        if (d.relu) v = fmaxf(v, 0.f);
        if (d.out) {
          v = rnd(d.out_dt, v);
          stv(d.out, d.out_dt, o, v);
        }
        if (d.stats) {
          n += 1.f;
          const float delta = v - mean;
          mean += delta / n;
          m2 = fmaf(delta, v - mean, m2);
        }
      }
    }
    if (d.stats) {
      if (rt.G == 1) {
        if (c < C) {
          d.stats[((int64_t)tile * C + c) * 2] = mean;
          d.stats[((int64_t)tile * C + c) * 2 + 1] = m2;
        }
      } else {
        red[threadIdx.x][0] = mean;
        red[threadIdx.x][1] = m2;
        __syncthreads();
        if ((int)threadIdx.x < C) {
          float a = 0.f, am = 0.f, a2 = 0.f;
          for (int g = 0; g < rt.G; ++g) {
            // rows r0 + g, r0 + g + G, ... below r1
            const float cg = r1 > r0 + g ? (float)((r1 - r0 - g + rt.G - 1) / rt.G) : 0.f;
            chan_merge(a, am, a2, cg, red[g * C + threadIdx.x][0], red[g * C + threadIdx.x][1]);
          }
          d.stats[((int64_t)tile * C + threadIdx.x) * 2] = am;
          d.stats[((int64_t)tile * C + threadIdx.x) * 2 + 1] = a2;
        }
        __syncthreads();
      }
    }
  }
}

__global__ void __launch_bounds__(256) k_ew_bwd(const EwBwdDesc* __restrict__ tab, const int* __restrict__ tstart,
                                                int n) {
  const int inst = find_instance(tstart, n, blockIdx.x);
  const EwBwdDesc& d = tab[inst];
  const int tile = blockIdx.x - tstart[inst];
  const int64_t base = (int64_t)tile * d.rows_per_tile * d.C;
  const int64_t end = min((int64_t)d.M * d.C, base + (int64_t)d.rows_per_tile * d.C);
  for (int64_t o = base + threadIdx.x; o < end; o += blockDim.x) {
    float g = d.dout[o];
    if (d.relu && !(ldv(d.out, d.out_dt, o) > 0.f)) g = 0.f;
    for (int i = 0; i < d.nin; ++i) {
      float v = d.coef[i] * g;
      d.gin[i][o] = d.acc[i] ? d.gin[i][o] + v : v;
    }
  }
}

// ---------------------------------------------------------------- BN
// one CTA per channel: thread t sums tiles t, t+256, ... in double, then a
// fixed shared-memory tree combines the 256 partial sums

// Sums over one chunk of partial tiles ([tiles][C][2] floats) for the 32
// channels of a channel group: lane = channel, warp w adds tiles t0+w, t0+w+8,
// ... (eight independent 256-byte row loads per warp), then warp 0 adds the
// eight warps' sums in warp order.  When a launch spans several chunks, each
// CTA leaves its chunk sums in scratch and the last CTA of the channel group
// (an atomic count) adds them: warp w takes chunks w, w+8, ..., warp 0 adds the
// warps' sums in order, so the result does not depend on the order the CTAs
// run in.  Returns true on the threads (warp 0, c < C) that hold the totals in
// s1 / s2.
__device__ __forceinline__ bool chunked_sums(const float* __restrict__ part, int C, int tiles, int cg, int chunk,
                                             int nchunk, double* scratch, int32_t* counter, double& s1, double& s2) {
  __shared__ double red[8][2][32];
  __shared__ int is_last;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int c = cg * 32 + lane;
  const int t0 = chunk * kFinTilesPerCta, t1 = min(tiles, t0 + kFinTilesPerCta);
  double a = 0.0, b = 0.0;
  if (c < C) {
    float2 v[kFinTilesPerCta / 8];
#pragma unroll
    for (int k = 0; k < kFinTilesPerCta / 8; ++k) {
      const int t = t0 + w + 8 * k;
      v[k] = t < t1 ? *reinterpret_cast<const float2*>(part + ((int64_t)t * C + c) * 2) : make_float2(0.f, 0.f);
    }
#pragma unroll
    for (int k = 0; k < kFinTilesPerCta / 8; ++k) {
      a += (double)v[k].x;
      b += (double)v[k].y;
    }
  }
  red[w][0][lane] = a;
  red[w][1][lane] = b;
  __syncthreads();
  a = 0.0;
  b = 0.0;
  if (w == 0)
    for (int k = 0; k < 8; ++k) {
      a += red[k][0][lane];
      b += red[k][1][lane];
    }
  if (nchunk == 1) {
    s1 = a;
    s2 = b;
    return w == 0 && c < C;
  }
  if (w == 0 && c < C) {
    scratch[((int64_t)chunk * C + c) * 2] = a;
    scratch[((int64_t)chunk * C + c) * 2 + 1] = b;
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) is_last = atomicAdd(counter + cg, 1) == nchunk - 1;
  __syncthreads();
  if (!is_last) return false;
  __threadfence();
  a = 0.0;
  b = 0.0;
  if (c < C)
    for (int k = w; k < nchunk; k += 8) {
      a += __ldcg(scratch + ((int64_t)k * C + c) * 2);
      b += __ldcg(scratch + ((int64_t)k * C + c) * 2 + 1);
    }
  red[w][0][lane] = a;
  red[w][1][lane] = b;
  __syncthreads();
  a = 0.0;
  b = 0.0;
  if (w == 0)
    for (int k = 0; k < 8; ++k) {
      a += red[k][0][lane];
      b += red[k][1][lane];
    }
  if (threadIdx.x == 0) counter[cg] = 0;  // ready for the next launch
  s1 = a;
  s2 = b;
  return w == 0 && c < C;
}

// The same two-level reduction for the forward statistics.  Partial tiles
// hold (mean_t, M2_t) of their rows (count n_t: rpt rows each, the last tile
// the remainder of M).  They are combined as shifted sums around K = mean_0
// (the first tile's mean, read by every CTA): with d_t = mean_t - K,
//   S1 = sum n_t d_t,   S2 = sum (M2_t + n_t d_t^2),
//   mean = K + S1 / M,  M2 = S2 - S1^2 / M,
// which is Chan's pairwise update written for many sets at once (no term
// subtracts two large sums: K lies within a few standard errors of the mean,
// so S1^2 / M is a small part of S2).  Plain fp64 sums in the fixed order of
// chunked_sums; returns true on the threads that hold (M, mean, M2).
__device__ __forceinline__ bool chunked_moments(const float* __restrict__ part, int C, int tiles, int64_t M, int rpt,
                                                int cg, int chunk, int nchunk, double* scratch, int32_t* counter,
                                                double& n_out, double& mean_out, double& m2_out) {
  __shared__ double red[8][2][32];
  __shared__ int is_last;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int c = cg * 32 + lane;
  const int t0 = chunk * kFinTilesPerCta, t1 = min(tiles, t0 + kFinTilesPerCta);
  double a = 0.0, b = 0.0;
  const float K = c < C && tiles > 0 ? __ldg(part + (int64_t)c * 2) : 0.f;
  if (c < C) {
    float2 v[kFinTilesPerCta / 8];
#pragma unroll
    for (int k = 0; k < kFinTilesPerCta / 8; ++k) {
      const int t = t0 + w + 8 * k;
      v[k] = t < t1 ? *reinterpret_cast<const float2*>(part + ((int64_t)t * C + c) * 2) : make_float2(0.f, 0.f);
    }
    // this thread's eight tiles in fp32 (d is a small difference of two
    // close means; the S2 terms are all positive), then fp64 from here on
    float fa = 0.f, fb = 0.f;
#pragma unroll
    for (int k = 0; k < kFinTilesPerCta / 8; ++k) {
      const int64_t t = t0 + w + 8 * k;
      if (t < t1) {
        const int64_t r1 = (t + 1) * rpt < M ? (t + 1) * rpt : M;
        const float n = (float)(r1 - t * rpt);
        const float d = v[k].x - K;
        const float nd = n * d;
        fa += nd;
        fb += v[k].y + nd * d;
      }
    }
    a = fa;
    b = fb;
  }
  red[w][0][lane] = a;
  red[w][1][lane] = b;
  __syncthreads();
  a = 0.0;
  b = 0.0;
  if (w == 0)
    for (int k = 0; k < 8; ++k) {
      a += red[k][0][lane];
      b += red[k][1][lane];
    }
  bool have = w == 0 && c < C;
  if (nchunk > 1) {
    if (w == 0 && c < C) {
      scratch[((int64_t)chunk * C + c) * 2] = a;
      scratch[((int64_t)chunk * C + c) * 2 + 1] = b;
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) is_last = atomicAdd(counter + cg, 1) == nchunk - 1;
    __syncthreads();
    if (!is_last) return false;
    __threadfence();
    a = 0.0;
    b = 0.0;
    if (c < C)
      for (int k = w; k < nchunk; k += 8) {
        a += __ldcg(scratch + ((int64_t)k * C + c) * 2);
        b += __ldcg(scratch + ((int64_t)k * C + c) * 2 + 1);
      }
    __syncthreads();  // warp 0 has read red[] of the chunk pass
    red[w][0][lane] = a;
    red[w][1][lane] = b;
    __syncthreads();
    a = 0.0;
    b = 0.0;
    if (w == 0)
      for (int k = 0; k < 8; ++k) {
        a += red[k][0][lane];
        b += red[k][1][lane];
      }
    if (threadIdx.x == 0) counter[cg] = 0;  // ready for the next launch
  }
  // one fp64 division (the reciprocal of the count); this part's fp64 units
  // are slow, and the callers finish in fp32
  const double n = (double)M;
  const double rn = 1.0 / n;
  n_out = n;
  mean_out = (double)K + a * rn;
  m2_out = b - a * a * rn;
  return have;
}

__global__ void __launch_bounds__(256) k_bn_fin(const BnFinDesc* __restrict__ tab, const int* __restrict__ tstart,
                                                int n) {
  const int inst = find_instance(tstart, n, blockIdx.x);
  const BnFinDesc& d = tab[inst];
  const int local = blockIdx.x - tstart[inst];
  const int cg = local % d.cgroups, chunk = local / d.cgroups;
  const int c = cg * 32 + (threadIdx.x & 31);
  float mean, var;
  if (d.eval) {
    // eval mode: the running statistics stand in for the batch's
    if (threadIdx.x >= 32 || c >= d.C) return;
    mean = d.run_mean[c];
    var = d.run_var[c];
  } else {
    double cnt, mean64, m2;
    if (!chunked_moments(d.part, d.C, d.tiles, d.count, d.rows_per_tile, cg, chunk, d.nchunk, d.scratch, d.counter,
                         cnt, mean64, m2))
      return;
    // (the sums were fp64; from here fp32 holds every quantity to 2^-24)
    mean = (float)mean64;
    var = cnt > 0.0 ? (float)m2 / (float)cnt : 0.f;
    if (var < 0.f) var = 0.f;
    if (d.run_mean) {
      // running statistics follow the batch mean and the unbiased variance
      const float m = d.momentum;
      const float unbiased = d.count > 1 ? var * ((float)d.count / (float)(d.count - 1)) : var;
      d.run_mean[c] = (1.f - m) * d.run_mean[c] + m * mean;
      d.run_var[c] = (1.f - m) * d.run_var[c] + m * unbiased;
    }
  }
  const float rstd = 1.f / sqrtf(var + 1e-5f);
  const float sc = d.gamma[c] * rstd;
  d.mean[c] = mean;
  d.rstd[c] = rstd;
  d.scale[c] = sc;
  d.shift[c] = fmaf(-mean, sc, d.beta[c]);
}

__global__ void __launch_bounds__(256) k_bnb_reduce(const BnBwdDesc* __restrict__ tab,
                                                    const int* __restrict__ tstart, int n) {
  __shared__ float red[256][2];
  const int inst = find_instance(tstart, n, blockIdx.x);
  const BnBwdDesc& d = tab[inst];
  const int tile = blockIdx.x - tstart[inst];
  const int C = d.C;
  const RowTile rt(C, threadIdx.x);
  const int64_t r0 = (int64_t)tile * d.rows_per_tile;
  const int64_t r1 = min((int64_t)d.M, r0 + d.rows_per_tile);
  for (int ci = 0; ci < rt.cpt; ++ci) {
    const int c = rt.c0 + 256 * ci;
    float s1 = 0.f, s2 = 0.f;
    if (c < C) {
      const float mean = d.mean[c], rstd = d.rstd[c], sc = d.scale[c], sh = d.shift[c];
      for (int64_t r = r0 + rt.g; r < r1; r += rt.G) {
        const int64_t o = r * C + c;
        const float h = ldv(d.h, d.h_dt, o);
        float dz = d.da[o];
        if (d.relu && !(fmaf(sc, h, sh) > 0.f)) dz = 0.f;
        s1 += dz;
        s2 += dz * ((h - mean) * rstd);
      }
    }
    if (rt.G == 1) {
      if (c < C) {
        d.part[((int64_t)tile * C + c) * 2] = s1;
        d.part[((int64_t)tile * C + c) * 2 + 1] = s2;
      }
    } else {
      red[threadIdx.x][0] = s1;
      red[threadIdx.x][1] = s2;
      __syncthreads();
      if ((int)threadIdx.x < C) {
        float a = 0.f, b = 0.f;
        for (int g = 0; g < rt.G; ++g) { a += red[g * C + threadIdx.x][0]; b += red[g * C + threadIdx.x][1]; }
        d.part[((int64_t)tile * C + threadIdx.x) * 2] = a;
        d.part[((int64_t)tile * C + threadIdx.x) * 2 + 1] = b;
      }
      __syncthreads();
    }
  }
}

__global__ void __launch_bounds__(256) k_bnb_fin(const BnBwdDesc* __restrict__ tab, const int* __restrict__ tstart,
                                                 int n) {
  const int inst = find_instance(tstart, n, blockIdx.x);
  const BnBwdDesc& d = tab[inst];
  const int local = blockIdx.x - tstart[inst];
  const int cg = local % d.cgroups, chunk = local / d.cgroups;
  const int c = cg * 32 + (threadIdx.x & 31);
  double s1, s2;
  if (!chunked_sums(d.part, d.C, d.tiles, cg, chunk, d.nchunk, d.scratch, d.counter, s1, s2)) return;
  d.dbeta[c] = d.accumulate ? d.dbeta[c] + (float)s1 : (float)s1;
  d.dgamma[c] = d.accumulate ? d.dgamma[c] + (float)s2 : (float)s2;
  d.coef[c * 3 + 0] = d.gamma[c] * d.rstd[c];
  const double rm = 1.0 / (double)d.M;
  d.coef[c * 3 + 1] = (float)(s1 * rm);
  d.coef[c * 3 + 2] = (float)(s2 * rm);
}

__global__ void __launch_bounds__(256) k_bnb_apply(const BnBwdDesc* __restrict__ tab,
                                                   const int* __restrict__ tstart, int n) {
  const int inst = find_instance(tstart, n, blockIdx.x);
  const BnBwdDesc& d = tab[inst];
  const int tile = blockIdx.x - tstart[inst];
  const int C = d.C;
  const int64_t base = (int64_t)tile * d.rows_per_tile * C;
  const int64_t end = min((int64_t)d.M * C, base + (int64_t)d.rows_per_tile * C);
  for (int64_t o = base + threadIdx.x; o < end; o += blockDim.x) {
    const int c = (int)(o % C);
    const float h = ldv(d.h, d.h_dt, o);
    float dz = d.da[o];
    if (d.relu && !(fmaf(d.scale[c], h, d.shift[c]) > 0.f)) dz = 0.f;
    const float xhat = (h - d.mean[c]) * d.rstd[c];
    float v = d.coef[c * 3] * (dz - d.coef[c * 3 + 1] - xhat * d.coef[c * 3 + 2]);
    if (d.add0) v = fmaf(d.add_c[0], d.add0[o], v);
    if (d.add1) v = fmaf(d.add_c[1], d.add1[o], v);
    d.dh[o] = d.accumulate ? d.dh[o] + v : v;
  }
}

// ---------------------------------------------------------------- BN backward, 8 channels per thread
// Used when C % 8 == 0: each thread moves 8 consecutive channels of one row
// with 16/32-byte accesses.
__device__ __forceinline__ void ld8f(const float* p, float* v) {
  const float4 a = *reinterpret_cast<const float4*>(p), b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void st8f(float* p, const float* v) {
  *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  *reinterpret_cast<float4*>(p + 4) = make_float4(v[4], v[5], v[6], v[7]);
}
__device__ __forceinline__ void ld8any(const void* base, int dt, int64_t i, float* v) {
  if (dt == DT_F32) {
    ld8f(reinterpret_cast<const float*>(base) + i, v);
  } else {
    const uint4 u = *reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(base) + i);
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 f = __bfloat1622float2(h[k]);
      v[2 * k] = f.x;
      v[2 * k + 1] = f.y;
    }
  }
}

__global__ void __launch_bounds__(256) k_bnb_reduce8(const BnBwdDesc* __restrict__ tab,
                                                     const int* __restrict__ tstart, int n) {
  __shared__ float red[16][256];  // [quantity x channel][thread]: a warp touches 32 consecutive words
  const int inst = find_instance(tstart, n, blockIdx.x);
  const BnBwdDesc d = tab[inst];
  const int tile = blockIdx.x - tstart[inst];
  const int C = d.C, CG = C / 8;
  const int G = 256 / CG;  // row groups (CG <= 256)
  const int cg = threadIdx.x % CG, g = threadIdx.x / CG;
  const int64_t r0 = (int64_t)tile * d.rows_per_tile;
  const int64_t r1 = min((int64_t)d.M, r0 + d.rows_per_tile);
  float s1[8], s2[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) { s1[k] = 0.f; s2[k] = 0.f; }
  if (g < G) {
    const int c0 = cg * 8;
    float mean[8], rstd[8], sc[8], sh[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      mean[k] = d.mean[c0 + k]; rstd[k] = d.rstd[c0 + k]; sc[k] = d.scale[c0 + k]; sh[k] = d.shift[c0 + k];
    }
    for (int64_t r = r0 + g; r < r1; r += G) {
      const int64_t o = r * C + c0;
      float h[8], dz[8];
      ld8any(d.h, d.h_dt, o, h);
      ld8f(d.da + o, dz);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        if (d.relu && !(fmaf(sc[k], h[k], sh[k]) > 0.f)) dz[k] = 0.f;
        s1[k] += dz[k];
        s2[k] += dz[k] * ((h[k] - mean[k]) * rstd[k]);
      }
    }
  }
#pragma unroll
  for (int k = 0; k < 8; ++k) { red[k][threadIdx.x] = s1[k]; red[8 + k][threadIdx.x] = s2[k]; }
  __syncthreads();
  int groups = G;
  if ((G & (G - 1)) == 0) {
    // tree over the row groups: red[.][g * CG + cg] += red[.][(g + st) * CG + cg]
    for (int st = G >> 1; st > 0; st >>= 1) {
      if (g < st) {
#pragma unroll
        for (int k = 0; k < 16; ++k) red[k][threadIdx.x] += red[k][threadIdx.x + st * CG];
      }
      __syncthreads();
    }
    groups = 1;
  }
  if ((int)threadIdx.x < CG) {
    float a[8], b[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) { a[k] = 0.f; b[k] = 0.f; }
    for (int gg = 0; gg < groups; ++gg)
#pragma unroll
      for (int k = 0; k < 8; ++k) { a[k] += red[k][gg * CG + threadIdx.x]; b[k] += red[8 + k][gg * CG + threadIdx.x]; }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      d.part[((int64_t)tile * C + threadIdx.x * 8 + k) * 2] = a[k];
      d.part[((int64_t)tile * C + threadIdx.x * 8 + k) * 2 + 1] = b[k];
    }
  }
}

// Each thread keeps one group of 8 channels (cg = thread % (C/8)) for the
// whole tile, with that group's per-channel parameters in registers, and
// walks the tile's rows G = 256 / (C/8) apart.
__global__ void __launch_bounds__(256) k_bnb_apply8(const BnBwdDesc* __restrict__ tab,
                                                    const int* __restrict__ tstart, int n) {
  const int inst = find_instance(tstart, n, blockIdx.x);
  const BnBwdDesc d = tab[inst];  // a private copy: the stores below cannot force reloads
  const int tile = blockIdx.x - tstart[inst];
  const int C = d.C, CG = C / 8;
  const int G = 256 / CG;
  const int cg = threadIdx.x % CG, g = threadIdx.x / CG;
  if (g >= G) return;
  const int c0 = cg * 8;
  float sc[8], sh[8], mean[8], rstd[8], k0[8], k1[8], k2[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    sc[k] = d.scale[c0 + k]; sh[k] = d.shift[c0 + k]; mean[k] = d.mean[c0 + k]; rstd[k] = d.rstd[c0 + k];
    k0[k] = d.coef[(c0 + k) * 3]; k1[k] = d.coef[(c0 + k) * 3 + 1]; k2[k] = d.coef[(c0 + k) * 3 + 2];
  }
  const int64_t r0 = (int64_t)tile * d.rows_per_tile;
  const int64_t r1 = min((int64_t)d.M, r0 + d.rows_per_tile);
  for (int64_t r = r0 + g; r < r1; r += G) {
    const int64_t o = r * C + c0;
    float h[8], dz[8], out[8];
    ld8any(d.h, d.h_dt, o, h);
    ld8f(d.da + o, dz);
    float a0[8], a1[8], ac[8];
    if (d.add0) ld8f(d.add0 + o, a0);
    if (d.add1) ld8f(d.add1 + o, a1);
    if (d.accumulate) ld8f(d.dh + o, ac);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      if (d.relu && !(fmaf(sc[k], h[k], sh[k]) > 0.f)) dz[k] = 0.f;
      const float xhat = (h[k] - mean[k]) * rstd[k];
      out[k] = k0[k] * (dz[k] - k1[k] - xhat * k2[k]);
      if (d.add0) out[k] = fmaf(d.add_c[0], a0[k], out[k]);
      if (d.add1) out[k] = fmaf(d.add_c[1], a1[k], out[k]);
      if (d.accumulate) out[k] += ac[k];
    }
    st8f(d.dh + o, out);
  }
}

// ---------------------------------------------------------------- pooling
__global__ void __launch_bounds__(256) k_pool_fwd(const PoolDesc* __restrict__ tab, const int* __restrict__ tstart,
                                                  int n) {
  const int inst = find_instance(tstart, n, blockIdx.x);
  const PoolDesc& d = tab[inst];
  const int64_t i = (int64_t)(blockIdx.x - tstart[inst]) * 256 + threadIdx.x;
  const int64_t total = (int64_t)d.B * d.P * d.Q * d.C;
  if (i >= total) return;
  const int c = (int)(i % d.C);
  int64_t t = i / d.C;
  const int q = (int)(t % d.Q); t /= d.Q;
  const int p = (int)(t % d.P);
  const int nb = (int)(t / d.P);
  float best = -INFINITY;
  for (int r = 0; r < d.k; ++r)
    for (int s = 0; s < d.k; ++s) {
      const int h = p * d.stride + r - d.pad, w = q * d.stride + s - d.pad;
      if (h < 0 || h >= d.H || w < 0 || w >= d.W) continue;
      const float v = ld_src(d.x, ((int64_t)(nb * d.H + h) * d.W + w) * d.C + c, c);
      if (v > best) best = v;
    }
  stv(d.y, d.y_dt, i, best);
}

// dx[n,h,w,c] (+)= sum over windows whose first maximum sits at (h,w) of dy
__global__ void __launch_bounds__(256) k_pool_bwd(const PoolDesc* __restrict__ tab, const int* __restrict__ tstart,
                                                  int n) {
  const int inst = find_instance(tstart, n, blockIdx.x);
  const PoolDesc& d = tab[inst];
  const int64_t i = (int64_t)(blockIdx.x - tstart[inst]) * 256 + threadIdx.x;
  const int64_t total = (int64_t)d.B * d.H * d.W * d.C;
  if (i >= total) return;
  const int c = (int)(i % d.C);
  int64_t t = i / d.C;
  const int w = (int)(t % d.W); t /= d.W;
  const int h = (int)(t % d.H);
  const int nb = (int)(t / d.H);
  float g = 0.f;
  const int p_lo = max(0, (h + d.pad - d.k + d.stride) / d.stride), p_hi = min(d.P - 1, (h + d.pad) / d.stride);
  const int q_lo = max(0, (w + d.pad - d.k + d.stride) / d.stride), q_hi = min(d.Q - 1, (w + d.pad) / d.stride);
  for (int p = p_lo; p <= p_hi; ++p)
    for (int q = q_lo; q <= q_hi; ++q) {
      if (h + d.pad - p * d.stride >= d.k || w + d.pad - q * d.stride >= d.k) continue;
      float best = -INFINITY;
      int bh = -1, bw = -1;
      for (int r = 0; r < d.k; ++r)
        for (int s = 0; s < d.k; ++s) {
          const int hh = p * d.stride + r - d.pad, ww = q * d.stride + s - d.pad;
          if (hh < 0 || hh >= d.H || ww < 0 || ww >= d.W) continue;
          const float v = ld_src(d.x, ((int64_t)(nb * d.H + hh) * d.W + ww) * d.C + c, c);
          if (v > best) { best = v; bh = hh; bw = ww; }
        }
      if (bh == h && bw == w) g += d.dy[((int64_t)(nb * d.P + p) * d.Q + q) * d.C + c];
    }
  d.dx[i] = d.accumulate ? d.dx[i] + g : g;
}

// ---------------------------------------------------------------- GEMM (head)
// C[m][n] = sum_k A[m][k] B[k][n] (+ bias[n]) (+ beta C[m][n]) (ReLU), fp32.
// 64 x 64 tiles, 256 threads with 4 x 4 outputs each; the K loop runs in 32-wide
// steps with the next step's operands loaded into registers while the current
// one is multiplied from shared memory (double buffered).  Each operand is read
// along whichever of its two indices is contiguous in memory, so every warp load
// is coalesced for any of the head's layouts.  Every output sums its k terms in
// ascending order with one fused multiply-add each.
__global__ void __launch_bounds__(256) k_gemm(const GemmDesc* __restrict__ tab, const int* __restrict__ tstart,
                                              int n) {
  constexpr int BM = 64, BN = 64, BK = 32, PER = BM * BK / 256;
  __shared__ float As[2][BK][BM + 4];
  __shared__ float Bs[2][BK][BN + 4];
  const int inst = find_instance(tstart, n, blockIdx.x);
  const GemmDesc& d = tab[inst];
  const int t = blockIdx.x - tstart[inst];
  const int tm = t % d.mtiles, tn = t / d.mtiles;
  const int m0 = tm * BM, n0 = tn * BN;
  const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
  const bool a_k = d.sak == 1, b_k = d.sbk == 1;  // k contiguous in A / in B
  float ra[PER], rb[PER];
  auto slot = [&](int e, bool k_fast, int W, int& kk, int& x) {
    if (k_fast) { kk = e % BK; x = e / BK; } else { x = e % W; kk = e / W; }
  };
  auto load = [&](int k0) {
#pragma unroll
    for (int q = 0; q < PER; ++q) {
      int kk, x;
      slot(tid + 256 * q, a_k, BM, kk, x);
      const int m = m0 + x, k = k0 + kk;
      ra[q] = (m < d.M && k < d.K) ? d.A[(int64_t)m * d.sam + (int64_t)k * d.sak] : 0.f;
      slot(tid + 256 * q, b_k, BN, kk, x);
      const int nc = n0 + x, kb = k0 + kk;
      rb[q] = (nc < d.N && kb < d.K) ? d.Bm[(int64_t)kb * d.sbk + (int64_t)nc * d.sbn] : 0.f;
    }
  };
  auto store = [&](int buf) {
#pragma unroll
    for (int q = 0; q < PER; ++q) {
      int kk, x;
      slot(tid + 256 * q, a_k, BM, kk, x);
      As[buf][kk][x] = ra[q];
      slot(tid + 256 * q, b_k, BN, kk, x);
      Bs[buf][kk][x] = rb[q];
    }
  };
  float acc[4][4] = {};
  load(0);
  store(0);
  __syncthreads();
  int buf = 0;
  for (int k0 = 0; k0 < d.K; k0 += BK) {
    const bool more = k0 + BK < d.K;
    if (more) load(k0 + BK);
#pragma unroll
    for (int kk = 0; kk < BK; ++kk)
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(As[buf][kk][ty + 16 * i], Bs[buf][kk][tx + 16 * j], acc[i][j]);
    if (more) store(buf ^ 1);
    __syncthreads();
    buf ^= 1;
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int m = m0 + ty + 16 * i, nc = n0 + tx + 16 * j;
      if (m < d.M && nc < d.N) {
        float v = acc[i][j];
        if (d.bias) v += d.bias[nc];
        if (d.beta != 0.f) v += d.beta * d.Cm[(int64_t)m * d.scm + nc];
        if (d.relu) v = fmaxf(v, 0.f);
        d.Cm[(int64_t)m * d.scm + nc] = v;
      }
    }
}

// ---------------------------------------------------------------- head + misc
__global__ void k_gap(Src x, float* feat, int B, int HW, int C) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= B * C) return;
  const int b = i / C, c = i % C;
  float s = 0.f;
  for (int k = 0; k < HW; ++k) s += ld_src(x, ((int64_t)b * HW + k) * C + c, c);
  feat[i] = s / (float)HW;
}

__global__ void k_gap_bwd(const float* dfeat, float* dx, int B, int HW, int C) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)B * HW * C) return;
  const int c = (int)(i % C);
  const int b = (int)(i / ((int64_t)HW * C));
  dx[i] = dfeat[b * C + c] / (float)HW;
}

// one CTA: per-sample log-sum-exp loss, mean over the batch in a fixed order
__global__ void __launch_bounds__(256) k_softmax_ce(const float* logits, const int32_t* labels, int B, int m,
                                                    float* loss, float* dlogits, int32_t* status) {
  __shared__ float per[1024];
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  for (int b = warp; b < B; b += 8) {
    const float* z = logits + (int64_t)b * m;
    float mx = -INFINITY;
    for (int i = lane; i < m; i += 32) mx = fmaxf(mx, z[i]);
    for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    float se = 0.f;
    for (int i = lane; i < m; i += 32) se += expf(z[i] - mx);
    for (int off = 16; off > 0; off >>= 1) se += __shfl_xor_sync(0xffffffffu, se, off);
    const int lab = labels[b];
    const float lse = logf(se) + mx;
    for (int i = lane; i < m; i += 32) {
      const float p = expf(z[i] - mx) / se;
      dlogits[(int64_t)b * m + i] = (p - (i == lab ? 1.f : 0.f)) / (float)B;
    }
    if (lane == 0) per[b] = lse - ((lab >= 0 && lab < m) ? z[lab] : 0.f);
    if (lane == 0 && (lab < 0 || lab >= m)) atomicExch(status, 1);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int b = 0; b < B; ++b) s += per[b];
    const float l = (float)(s / B);
    *loss = l;
    if (!isfinite(l)) atomicExch(status, 2);
  }
}

__global__ void k_colsum(const float* A, int rows, int cols, float* out) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= cols) return;
  float s = 0.f;
  for (int r = 0; r < rows; ++r) s += A[(int64_t)r * cols + c];
  out[c] = s;
}

__global__ void k_relu_mask(float* g, const float* pre, int64_t n) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n && !(pre[i] > 0.f)) g[i] = 0.f;
}

__global__ void k_sgd(float* __restrict__ w, const float* __restrict__ g, float* __restrict__ v, void* shadow,
                      int32_t shadow_dt, int64_t n, float lr, float mu, float wd, int nesterov, int first) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    const float wi = w[i];
    const float di = fmaf(wd, wi, g[i]);
    const float vi = first ? di : fmaf(mu, v[i], di);
    v[i] = vi;
    const float step = nesterov ? fmaf(mu, vi, di) : vi;
    const float wn = fmaf(-lr, step, wi);
    w[i] = wn;
    if (shadow) stv(shadow, shadow_dt, i, wn);
  }
}

__global__ void k_pack_input(const float* x, void* out, int32_t dt, int B, int C, int H, int W) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t total = (int64_t)B * C * H * W;
  if (i >= total) return;
  const int c = (int)(i % C);
  int64_t t = i / C;
  const int w = (int)(t % W); t /= W;
  const int h = (int)(t % H);
  const int b = (int)(t / H);
  stv(out, dt, i, x[(((int64_t)b * C + c) * H + h) * W + w]);
}

__global__ void k_export(Src x, int B, int H, int W, int C, float* out) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t total = (int64_t)B * C * H * W;
  if (i >= total) return;
  const int c = (int)(i % C);
  int64_t t = i / C;
  const int w = (int)(t % W); t /= W;
  const int h = (int)(t % H);
  const int b = (int)(t / H);
  out[(((int64_t)b * C + c) * H + h) * W + w] = ld_src(x, i, c);
}

__global__ void k_copy_cast(const float* in, void* out, int32_t dt, int64_t n) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) stv(out, dt, i, in[i]);
}

// ---------------------------------------------------------------- launchers
static inline int cdiv64(int64_t a, int64_t b) { return (int)((a + b - 1) / b); }

namespace {
constexpr int kMaxDevices = 64;
std::atomic<int> g_sms[kMaxDevices];
std::atomic<uint32_t> g_attr_done[kMaxDevices];
std::mutex g_attr_mu;
}  // namespace

int device_sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 1;
  int v = g_sms[dev].load(std::memory_order_acquire);
  if (v > 0) return v;
  int sms = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) return 1;
  g_sms[dev].store(sms, std::memory_order_release);
  return sms;
}

cudaError_t set_smem_attr_once(int slot, const void* kernel, int bytes) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices || slot < 0 || slot >= 32) return cudaErrorInvalidValue;
  const uint32_t bit = 1u << slot;
  if (g_attr_done[dev].load(std::memory_order_acquire) & bit) return cudaSuccess;
  std::lock_guard<std::mutex> lk(g_attr_mu);
  if (g_attr_done[dev].load(std::memory_order_acquire) & bit) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) g_attr_done[dev].fetch_or(bit, std::memory_order_release);
  return e;
}

cudaError_t launch_conv_fwd_simt(const ConvDesc* tab, const int* tstart, int n, int total, int variant,
                                 cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  if (variant == 0) k_conv_fwd<64, 64><<<total, 256, 0, st>>>(tab, tstart, n);
  else if (variant == 1) k_conv_fwd<128, 32><<<total, 256, 0, st>>>(tab, tstart, n);
  else k_conv_fwd<256, 16><<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_conv_dgrad_simt(const ConvDesc* tab, const int* tstart, int n, int total, int variant,
                                   cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  if (variant == 0) k_conv_dgrad<64, 64><<<total, 256, 0, st>>>(tab, tstart, n);
  else if (variant == 1) k_conv_dgrad<128, 32><<<total, 256, 0, st>>>(tab, tstart, n);
  else k_conv_dgrad<256, 16><<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_conv_wgrad_simt(const ConvDesc* tab, const int* tstart, int n, int total, int variant,
                                   cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  if (variant == 1) k_conv_wgrad_small<<<total, 256, 0, st>>>(tab, tstart, n);
  else k_conv_wgrad<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_wreduce(const WReduceDesc* tab, const int* tstart, int n, int total, cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  k_wreduce<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_wtrans(const WtDesc* tab, const int* tstart, int n, int total, cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  k_wtrans<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_ew(const EwDesc* tab, const int* tstart, int n, int total, cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  k_ew<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_ew_bwd(const EwBwdDesc* tab, const int* tstart, int n, int total, cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  k_ew_bwd<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_bn_fin(const BnFinDesc* tab, const int* tstart, int n, int total, cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  k_bn_fin<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_bnb_reduce(const BnBwdDesc* tab, const int* tstart, int n, int total, cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  k_bnb_reduce<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_bnb_reduce8(const BnBwdDesc* tab, const int* tstart, int n, int total, cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  k_bnb_reduce8<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_bnb_fin(const BnBwdDesc* tab, const int* tstart, int n, int total, cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  k_bnb_fin<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_bnb_apply(const BnBwdDesc* tab, const int* tstart, int n, int total, cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  k_bnb_apply<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_bnb_apply8(const BnBwdDesc* tab, const int* tstart, int n, int total, cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  k_bnb_apply8<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_pool_fwd(const PoolDesc* tab, const int* tstart, int n, int total, cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  k_pool_fwd<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_pool_bwd(const PoolDesc* tab, const int* tstart, int n, int total, cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  k_pool_bwd<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_gemm(const GemmDesc* tab, const int* tstart, int n, int total, cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  k_gemm<<<total, 256, 0, st>>>(tab, tstart, n);
  return cudaGetLastError();
}
cudaError_t launch_pack_input(const float* x, void* out, int32_t dt, int B, int C, int H, int W, cudaStream_t st) {
  const int64_t total = (int64_t)B * C * H * W;
  k_pack_input<<<cdiv64(total, 256), 256, 0, st>>>(x, out, dt, B, C, H, W);
  return cudaGetLastError();
}
cudaError_t launch_gap(Src x, float* feat, int B, int HW, int C, cudaStream_t st) {
  k_gap<<<cdiv64((int64_t)B * C, 256), 256, 0, st>>>(x, feat, B, HW, C);
  return cudaGetLastError();
}
cudaError_t launch_gap_bwd(const float* dfeat, float* dx, int B, int HW, int C, cudaStream_t st) {
  k_gap_bwd<<<cdiv64((int64_t)B * HW * C, 256), 256, 0, st>>>(dfeat, dx, B, HW, C);
  return cudaGetLastError();
}
cudaError_t launch_softmax_ce(const float* logits, const int32_t* labels, int B, int m, float* loss,
                              float* dlogits, int32_t* status, cudaStream_t st) {
  if (B > 1024) return cudaErrorInvalidValue;
  k_softmax_ce<<<1, 256, 0, st>>>(logits, labels, B, m, loss, dlogits, status);
  return cudaGetLastError();
}
cudaError_t launch_colsum(const float* A, int rows, int cols, float* out, cudaStream_t st) {
  k_colsum<<<cdiv64(cols, 128), 128, 0, st>>>(A, rows, cols, out);
  return cudaGetLastError();
}
cudaError_t launch_relu_mask(float* g, const float* pre, int64_t n, cudaStream_t st) {
  k_relu_mask<<<cdiv64(n, 256), 256, 0, st>>>(g, pre, n);
  return cudaGetLastError();
}
cudaError_t launch_sgd(float* w, const float* g, float* v, void* shadow, int32_t shadow_dt, int64_t n, float lr,
                       float mu, float wd, int nesterov, int first, cudaStream_t st) {
  int blocks = cdiv64(n, 256);
  if (blocks > device_sm_count() * 16) blocks = device_sm_count() * 16;
  if (blocks < 1) blocks = 1;
  k_sgd<<<blocks, 256, 0, st>>>(w, g, v, shadow, shadow_dt, n, lr, mu, wd, nesterov, first);
  return cudaGetLastError();
}
cudaError_t launch_export(Src x, int B, int H, int W, int C, float* out, cudaStream_t st) {
  const int64_t total = (int64_t)B * C * H * W;
  k_export<<<cdiv64(total, 256), 256, 0, st>>>(x, B, H, W, C, out);
  return cudaGetLastError();
}
cudaError_t launch_copy_cast(const float* in, void* out, int32_t dt, int64_t n, cudaStream_t st) {
  int blocks = cdiv64(n, 256);
  if (blocks > device_sm_count() * 16) blocks = device_sm_count() * 16;
  if (blocks < 1) blocks = 1;
  k_copy_cast<<<blocks, 256, 0, st>>>(in, out, dt, n);
  return cudaGetLastError();
}
cudaError_t launch_weight_cast(const float* in, void* out, int32_t dt, int64_t n, cudaStream_t st) {
  return launch_copy_cast(in, out, dt, n, st);
}

}  // namespace pnn
