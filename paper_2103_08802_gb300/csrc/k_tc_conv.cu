// Grouped implicit-GEMM convolutions on the 5th-generation tensor cores
// (tcgen05.mma kind::f16: bf16 operands, fp32 accumulator in TMEM) for the
// fine subnetworks, the coarse blocks and the preprocessing convs of the
// parareal network: one launch covers the same layer of every subnetwork
// (Algorithm 1's parallel loop; Algorithm 2's parallel loop for the two
// gradient kernels).
//
//   forward  D[m = out pixel][n = k_out]   = sum_{k=(r,s,c)}     act(X)[pix(m,r,s)][c] * W[n][r][s][c]
//   dgrad    D[m = in pixel][n = c]        = sum_{k=(r,s,k_out)} dY[pix'(m,r,s)][k_out] * Wt[c][r][s][k_out]
//   wgrad    D[m = (r,s,c)][n = k_out]     = sum_{k = out pixel} act(X)[pix(k,r,s)][c] * dY[k][k_out]
//
// A tile is 128 rows (M) x all of N (<= 256, padded to a multiple of 16).  K
// streams through a ring of shared-memory stages, 64 bf16 per row per stage,
// in the 128-byte-swizzled K-major layout the MMA reads.  Warps 0-3 gather
// the operands (zero padding, BN scale/shift + ReLU of the producing layer on
// load, fp32 -> bf16), transposing 8x8 blocks in registers where the K index
// is the pixel (wgrad).  Warp 4 owns TMEM; one of its threads issues the MMAs
// and commits each stage back to the producers.  Warps 0-3 then read the
// accumulator rows they own (TMEM lanes 32w..32w+31) and run the epilogue:
// forward -- residual add, store, BN partial sums; dgrad -- store or
// accumulate dX; wgrad -- store the split's partial dW.
//
// Every wait is bounded (globaltimer); on expiry the CTA records status 3,
// stops issuing work, drains its committed MMAs (bounded) and frees its TMEM.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "pnn_internal.h"
#include "tc_ptx.cuh"

namespace pnn {

namespace {

using namespace tc;

constexpr int kStages = 4;
constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kABytes = kBM * kBK * 2;
constexpr int kThreads = 160;
enum { FWD = 0, DGRAD = 1, WGRAD = 2 };

struct Shared {
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t accum;
  uint32_t tmem;
  int abort_flag;
  float red[4][256][2];
};

__device__ __forceinline__ int find_inst(const int* tstart, int n, int b) {
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (__ldg(tstart + mid) <= b) lo = mid; else hi = mid - 1;
  }
  return lo;
}

}  // namespace

template <int MODE>
__global__ void __launch_bounds__(kThreads, 1) k_conv_tc(const ConvDesc* __restrict__ tab,
                                                         const int* __restrict__ tstart, int ninst, int bnmax,
                                                         int32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* const gbase = smem_raw + (base - raw);
  const int inst = find_inst(tstart, ninst, blockIdx.x);
  const ConvDesc& d = tab[inst];
  int t = blockIdx.x - tstart[inst];
  const int tm = t % d.mtiles;
  t /= d.mtiles;
  const int tn = t % d.ntiles;
  const int split = t / d.ntiles;
  // GEMM geometry of this instance
  const int Mrows = MODE == FWD ? d.B * d.P * d.Q : (MODE == DGRAD ? d.B * d.H * d.W : d.R * d.S * d.C);
  const int Ncols = MODE == DGRAD ? d.C : d.K;
  const int Kt = MODE == FWD ? d.R * d.S * d.C : (MODE == DGRAD ? d.R * d.S * d.K : 0);
  const int pbeg = MODE == WGRAD ? split * d.pix_per_split : 0;
  const int pend = MODE == WGRAD ? min(d.B * d.P * d.Q, pbeg + d.pix_per_split) : 0;
  const int nkt = MODE == WGRAD ? (pend - pbeg + kBK - 1) / kBK : (Kt + kBK - 1) / kBK;
  const int BN = d.ntiles == 1 ? ((Ncols + 15) & ~15) : 256;
  const int n0 = tn * 256;
  const int m0 = tm * kBM;
  const int stage_bytes = kABytes + bnmax * 128;
  Shared& sh = *reinterpret_cast<Shared*>(gbase + kStages * stage_bytes);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  uint32_t ncols = 32;
  while ((int)ncols < BN) ncols <<= 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_u32(&sh.full[s]), 128);
      mbar_init(smem_u32(&sh.empty[s]), 1);
    }
    mbar_init(smem_u32(&sh.accum), 1);
    sh.abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 4) tmem_alloc(smem_u32(&sh.tmem), ncols);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = sh.tmem;
  volatile int* abort_flag = &sh.abort_flag;

  if (warp < 4) {
    // ================================================= producers
    const int cc = threadIdx.x & 7;   // 16-byte chunk of the 128-byte row
    const int rg = threadIdx.x >> 3;  // rows rg + 16 i
    int pn[8], ph[8], pw[8];
    if (MODE != WGRAD) {
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int m = m0 + rg + 16 * i;
        pn[i] = -1; ph[i] = 0; pw[i] = 0;
        if (m < Mrows) {
          if (MODE == FWD) {
            const int q = m % d.Q, tmp = m / d.Q;
            pw[i] = q * d.stride - d.pad;
            ph[i] = (tmp % d.P) * d.stride - d.pad;
            pn[i] = tmp / d.P;
          } else {
            const int w = m % d.W, tmp = m / d.W;
            pw[i] = w + d.pad;
            ph[i] = (tmp % d.H) + d.pad;
            pn[i] = tmp / d.H;
          }
        }
      }
    }
    bool ok = true;
    for (int kt = 0; kt < nkt; ++kt) {
      const int s = kt % kStages;
      if (!mbar_wait(smem_u32(&sh.empty[s]), ((kt / kStages) & 1) ^ 1, abort_flag)) { ok = false; break; }
      uint8_t* A = gbase + s * stage_bytes;
      uint8_t* Bt = A + kABytes;
      if (MODE == FWD) {
        const int k = kt * kBK + cc * 8;
        const bool kin = k < Kt;
        int c0 = 0, r_ = 0, s_ = 0;
        if (kin) { c0 = k % d.C; const int rs = k / d.C; s_ = rs % d.S; r_ = rs / d.S; }
        float sc[8], sf[8];
        const bool tr = kin && d.x.scale != nullptr;
        if (tr) {
#pragma unroll
          for (int i = 0; i < 8; ++i) { sc[i] = __ldg(d.x.scale + c0 + i); sf[i] = __ldg(d.x.shift + c0 + i); }
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int row = rg + 16 * i;
          uint4 out = make_uint4(0, 0, 0, 0);
          if (kin && pn[i] >= 0) {
            const int h = ph[i] + r_, w = pw[i] + s_;
            if (h >= 0 && h < d.H && w >= 0 && w < d.W) {
              float v[8];
              load8(d.x.ptr, d.x.dt, ((int64_t)(pn[i] * d.H + h) * d.W + w) * d.C + c0, v);
              if (tr) {
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                  v[j] = fmaf(sc[j], v[j], sf[j]);
                  if (d.x.relu) v[j] = fmaxf(v[j], 0.f);
                }
              }
              out = pack8(v);
            }
          }
          *reinterpret_cast<uint4*>(A + swz(row, cc)) = out;
        }
      } else if (MODE == DGRAD) {
        const int k = kt * kBK + cc * 8;
        const bool kin = k < Kt;
        int ko0 = 0, r_ = 0, s_ = 0;
        if (kin) { ko0 = k % d.K; const int rs = k / d.K; s_ = rs % d.S; r_ = rs / d.S; }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int row = rg + 16 * i;
          uint4 out = make_uint4(0, 0, 0, 0);
          if (kin && pn[i] >= 0) {
            const int pn_ = ph[i] - r_, qn_ = pw[i] - s_;
            if (pn_ >= 0 && qn_ >= 0 && pn_ % d.stride == 0 && qn_ % d.stride == 0) {
              const int p = pn_ / d.stride, q = qn_ / d.stride;
              if (p < d.P && q < d.Q) {
                float v[8];
                load8(d.dy, 0, ((int64_t)(pn[i] * d.P + p) * d.Q + q) * d.K + ko0, v);
                out = pack8(v);
              }
            }
          }
          *reinterpret_cast<uint4*>(A + swz(row, cc)) = out;
        }
      } else {
        // A: rows j = (r,s,c), K = 64 output pixels; unit = 8 rows x 8 pixels
        const int pix0 = pbeg + kt * kBK;
        {
          const int jg = threadIdx.x >> 3, pg = threadIdx.x & 7;
          const int j0 = m0 + jg * 8;
          uint4 in[8];
          const bool jin = j0 < Mrows;
          int c0 = 0, r_ = 0, s_ = 0;
          if (jin) { c0 = j0 % d.C; const int rs = j0 / d.C; s_ = rs % d.S; r_ = rs / d.S; }
          float sc[8], sf[8];
          const bool tr = jin && d.x.scale != nullptr;
          if (tr) {
#pragma unroll
            for (int i = 0; i < 8; ++i) { sc[i] = __ldg(d.x.scale + c0 + i); sf[i] = __ldg(d.x.shift + c0 + i); }
          }
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            in[i] = make_uint4(0, 0, 0, 0);
            const int pix = pix0 + pg * 8 + i;
            if (jin && pix < pend) {
              const int q = pix % d.Q, tmp = pix / d.Q, p = tmp % d.P, nb = tmp / d.P;
              const int h = p * d.stride + r_ - d.pad, w = q * d.stride + s_ - d.pad;
              if (h >= 0 && h < d.H && w >= 0 && w < d.W) {
                float v[8];
                load8(d.x.ptr, d.x.dt, ((int64_t)(nb * d.H + h) * d.W + w) * d.C + c0, v);
                if (tr) {
#pragma unroll
                  for (int j = 0; j < 8; ++j) {
                    v[j] = fmaf(sc[j], v[j], sf[j]);
                    if (d.x.relu) v[j] = fmaxf(v[j], 0.f);
                  }
                }
                in[i] = pack8(v);
              }
            }
          }
          uint4 out[8];
          transpose8(in, out);
#pragma unroll
          for (int c = 0; c < 8; ++c) *reinterpret_cast<uint4*>(A + swz(jg * 8 + c, pg)) = out[c];
        }
        // B: rows k_out, K = 64 output pixels
        for (int idx = threadIdx.x; idx < BN; idx += 128) {
          const int kg = idx >> 3, pg = idx & 7;
          const int ko0 = n0 + kg * 8;
          uint4 in[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            in[i] = make_uint4(0, 0, 0, 0);
            const int pix = pix0 + pg * 8 + i;
            if (ko0 < d.K && pix < pend) {
              float v[8];
              load8(d.dy, 0, (int64_t)pix * d.K + ko0, v);
              in[i] = pack8(v);
            }
          }
          uint4 out[8];
          transpose8(in, out);
#pragma unroll
          for (int c = 0; c < 8; ++c) *reinterpret_cast<uint4*>(Bt + swz(kg * 8 + c, pg)) = out[c];
        }
      }
      if (MODE != WGRAD) {
        // B: weight rows (forward: W[n][k], dgrad: Wt[c][k]), K-contiguous
        for (int idx = threadIdx.x; idx < BN * 8; idx += 128) {
          const int n = idx >> 3, ch = idx & 7;
          const int kk = kt * kBK + ch * 8;
          uint4 v = make_uint4(0, 0, 0, 0);
          if (n0 + n < Ncols && kk < Kt) {
            const uint4* q = reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(d.w) +
                                                            (int64_t)(n0 + n) * Kt + kk);
            if (PNN_ALIGNED(q, 16)) v = __ldg(q);
          }
          *reinterpret_cast<uint4*>(Bt + swz(n, ch)) = v;
        }
      }
      fence_proxy_async();
      mbar_arrive(smem_u32(&sh.full[s]));
    }
    if (!ok) {
      sh.abort_flag = 1;
      atomicExch(status, 3);
    }
    // ================================================= epilogue
    bool got = ok && mbar_wait(smem_u32(&sh.accum), 0, abort_flag);
    if (!got && ok) { sh.abort_flag = 1; atomicExch(status, 3); }
    got = __all_sync(0xffffffffu, got);  // tcgen05.ld is warp-collective
    fence_after();
    const int row = warp * 32 + lane;
    const int m = m0 + row;
    const bool mvalid = m < Mrows;
    const uint32_t tbase = tmem + ((uint32_t)(warp * 32) << 16);
    for (int j0 = 0; j0 < BN; j0 += 16) {
      float v[16];
      if (got) tmem_ld16(tbase + j0, v);
      else
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = 0.f;
      const int nb = n0 + j0;
      const bool full = nb + 16 <= Ncols;
      if (MODE == FWD) {
        float s1[16], s2[16];
        if (mvalid && got) {
          const int64_t o = (int64_t)m * d.K + nb;
          const bool vec = full && (d.K % 8) == 0;
          if (d.res) {
            if (vec) {
              float r8[8];
              load8(d.res, d.res_dt == DT_BF16, o, r8);
#pragma unroll
              for (int i = 0; i < 8; ++i) v[i] += r8[i];
              load8(d.res, d.res_dt == DT_BF16, o + 8, r8);
#pragma unroll
              for (int i = 0; i < 8; ++i) v[8 + i] += r8[i];
            } else {
              for (int i = 0; i < 16 && nb + i < d.K; ++i)
                v[i] += d.res_dt == DT_F32 ? reinterpret_cast<const float*>(d.res)[o + i]
                                           : __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(d.res)[o + i]);
            }
          }
          if (d.y_dt == DT_BF16) {
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = __bfloat162float(__float2bfloat16_rn(v[i]));
          }
          if (vec && PNN_ALIGNED((d.y_dt == DT_BF16 ? (const void*)(reinterpret_cast<__nv_bfloat16*>(d.y) + o)
                                                     : (const void*)(reinterpret_cast<float*>(d.y) + o)), 16)) {
            if (d.y_dt == DT_BF16) {
              uint4* p = reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(d.y) + o);
              p[0] = pack8(v);
              p[1] = pack8(v + 8);
            } else {
              float4* p = reinterpret_cast<float4*>(reinterpret_cast<float*>(d.y) + o);
              p[0] = make_float4(v[0], v[1], v[2], v[3]);
              p[1] = make_float4(v[4], v[5], v[6], v[7]);
              p[2] = make_float4(v[8], v[9], v[10], v[11]);
              p[3] = make_float4(v[12], v[13], v[14], v[15]);
            }
          } else if (!vec) {
            for (int i = 0; i < 16 && nb + i < d.K; ++i) {
              if (d.y_dt == DT_BF16) reinterpret_cast<__nv_bfloat16*>(d.y)[o + i] = __float2bfloat16_rn(v[i]);
              else reinterpret_cast<float*>(d.y)[o + i] = v[i];
            }
          }
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const bool cin = nb + i < d.K;
            s1[i] = cin ? v[i] : 0.f;
            s2[i] = cin ? v[i] * v[i] : 0.f;
          }
        } else {
#pragma unroll
          for (int i = 0; i < 16; ++i) { s1[i] = 0.f; s2[i] = 0.f; }
        }
        if (d.stats) {
#pragma unroll
          for (int i = 0; i < 16; ++i) {
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
              s1[i] += __shfl_xor_sync(0xffffffffu, s1[i], off);
              s2[i] += __shfl_xor_sync(0xffffffffu, s2[i], off);
            }
          }
          if (lane == 0) {
#pragma unroll
            for (int i = 0; i < 16; ++i) { sh.red[warp][j0 + i][0] = s1[i]; sh.red[warp][j0 + i][1] = s2[i]; }
          }
        }
      } else if (mvalid && got) {
        // dgrad: dX[m][c] (+)= v; wgrad: part[split][j = m][k_out] = v
        float* out = MODE == DGRAD ? d.dx + (int64_t)m * d.C + nb
                                   : d.dw_part + ((int64_t)split * Mrows + m) * d.K + nb;
        const bool acc = MODE == DGRAD && d.accumulate;
        if (full && (Ncols % 4) == 0) {
          float4* p = reinterpret_cast<float4*>(out);
          if (!PNN_ALIGNED(p, 16)) continue;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            float4 a = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
            if (acc) {
              const float4 b = p[q];
              a.x += b.x; a.y += b.y; a.z += b.z; a.w += b.w;
            }
            p[q] = a;
          }
        } else {
          for (int i = 0; i < 16 && nb + i < Ncols; ++i) out[i] = acc ? out[i] + v[i] : v[i];
        }
      }
    }
    if (MODE == FWD && d.stats) {
      asm volatile("bar.sync 1, 128;" ::: "memory");
      for (int j = threadIdx.x; j < BN; j += 128) {
        if (n0 + j < d.K) {
          const float a = sh.red[0][j][0] + sh.red[1][j][0] + sh.red[2][j][0] + sh.red[3][j][0];
          const float b = sh.red[0][j][1] + sh.red[1][j][1] + sh.red[2][j][1] + sh.red[3][j][1];
          d.stats[((int64_t)tm * d.K + n0 + j) * 2] = a;
          d.stats[((int64_t)tm * d.K + n0 + j) * 2 + 1] = b;
        }
      }
    }
  } else if (lane == 0) {
    // ================================================= MMA issuer
    const uint32_t idesc = idesc_bf16(kBM, BN);
    bool ok = true;
    for (int kt = 0; kt < nkt; ++kt) {
      const int s = kt % kStages;
      if (!mbar_wait(smem_u32(&sh.full[s]), (kt / kStages) & 1, abort_flag)) { ok = false; break; }
      fence_after();
      const uint32_t a_addr = base + s * stage_bytes;
      const uint32_t b_addr = a_addr + kABytes;
      const int krem = MODE == WGRAD ? pend - (pbeg + kt * kBK) : Kt - kt * kBK;
      const int ksub = min(4, (krem + 15) / 16);
      for (int kk = 0; kk < ksub; ++kk)
        mma_bf16(tmem, sw128_desc(a_addr + kk * 32), sw128_desc(b_addr + kk * 32), idesc, (kt | kk) ? 1u : 0u);
      mma_commit(smem_u32(&sh.empty[s]));
    }
    if (ok) {
      mma_commit(smem_u32(&sh.accum));
    } else {
      sh.abort_flag = 1;
      atomicExch(status, 3);
      mma_commit(smem_u32(&sh.accum));
      mbar_wait_drain(smem_u32(&sh.accum), 0);
    }
  }
  fence_before();
  __syncthreads();
  if (warp == 4) {
    fence_after();
    tmem_dealloc(tmem, ncols);
  }
}

static size_t smem_bytes(int bnmax) { return 1024 + kStages * (kABytes + (size_t)bnmax * 128) + sizeof(Shared); }

template <int MODE>
static cudaError_t launch_mode(const ConvDesc* tab, const int* tstart, int n, int total, int bnmax, int32_t* status,
                               cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  if (bnmax < 16 || bnmax > 256 || (bnmax & 15)) return cudaErrorInvalidValue;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_conv_tc<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem_bytes(256));
    if (e != cudaSuccess) return e;
    attr = true;
  }
  k_conv_tc<MODE><<<total, kThreads, smem_bytes(bnmax), st>>>(tab, tstart, n, bnmax, status);
  return cudaGetLastError();
}

cudaError_t launch_conv_fwd_tc(const ConvDesc* tab, const int* tstart, int n, int total, int bnmax, int32_t* status,
                               cudaStream_t st) {
  return launch_mode<FWD>(tab, tstart, n, total, bnmax, status, st);
}
cudaError_t launch_conv_dgrad_tc(const ConvDesc* tab, const int* tstart, int n, int total, int bnmax,
                                 int32_t* status, cudaStream_t st) {
  return launch_mode<DGRAD>(tab, tstart, n, total, bnmax, status, st);
}
unsigned long long conv_tc_debug_word() {
#ifdef PNN_DEBUG_CHECKS
  unsigned long long v = 0;
  cudaMemcpyFromSymbol(&v, tc::g_dbg, sizeof v);
  return v;
#else
  return 0;
#endif
}

cudaError_t launch_conv_wgrad_tc(const ConvDesc* tab, const int* tstart, int n, int total, int bnmax,
                                 int32_t* status, cudaStream_t st) {
  return launch_mode<WGRAD>(tab, tstart, n, total, bnmax, status, st);
}

}  // namespace pnn
