// Grouped implicit-GEMM convolution on the 5th-generation tensor cores
// (tcgen05.mma kind::f16, bf16 x bf16 -> fp32 accumulator in TMEM) for the
// fine subnetworks, coarse blocks and preprocessing convs of the parareal
// network (Algorithm 1's parallel loop: one launch covers the same layer of
// every subnetwork).
//
// Tile: 128 output pixels (M) x all output channels (N <= 256, a multiple of
// 16) of one problem instance.  The reduction K = R*S*C (tap-major, channel
// fastest) streams through a ring of shared-memory stages, 64 bf16 per row
// per stage, in the 128-byte-swizzled K-major layout the MMA reads:
//   byte(row, chunk) = row*128 + ((chunk ^ (row & 7)) << 4)   (16-byte chunks)
// Warps 0-3 gather the im2col rows (zero padding, optional BN scale/shift +
// ReLU of the producing layer applied on load), convert to bf16 and write the
// swizzled rows; warp 4 owns the TMEM allocation and one of its threads issues
// the MMAs.  mbarriers hand stages back and forth; tcgen05.commit releases a
// stage when the MMAs reading it have completed.  After the last stage warps
// 0-3 read the accumulator rows they own (TMEM lanes 32w..32w+31), add the
// residual, round, store, and reduce per-channel BN partial sums.
//
// Every wait is bounded (globaltimer); on expiry the CTA records status 3 in
// the status word, stops issuing work, drains its committed MMAs (bounded) and
// frees its TMEM before returning.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "pnn_internal.h"

namespace pnn {

namespace {

constexpr int kStages = 4;
constexpr int kBM = 128;
constexpr int kBK = 64;                          // bf16 elements per row per stage (128 bytes)
constexpr int kABytes = kBM * kBK * 2;           // 16 KiB
constexpr int kThreads = 160;                    // 4 producer/epilogue warps + 1 MMA warp
constexpr unsigned long long kWaitNs = 2000000000ull;  // 2 s budget per wait

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ unsigned long long gtimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// bounded wait; false on timeout or when another thread of the CTA aborted
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  if (mbar_try(bar, parity)) return true;
  const unsigned long long t0 = gtimer();
  while (true) {
    if (mbar_try(bar, parity)) return true;
    if (*abort_flag) return false;
    if (gtimer() - t0 > kWaitNs) return false;
  }
}
// time-bounded wait that ignores the abort flag (used to drain committed MMAs)
__device__ __forceinline__ bool mbar_wait_drain(uint32_t bar, uint32_t parity) {
  const unsigned long long t0 = gtimer();
  while (!mbar_try(bar, parity))
    if (gtimer() - t0 > kWaitNs) return false;
  return true;
}
__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups 1024 B apart
__device__ __forceinline__ uint64_t sw128_desc(uint32_t addr) {
  uint64_t d = 0;
  d |= (uint64_t)((addr & 0x3FFFF) >> 4);          // start address
  d |= (uint64_t)1 << 16;                          // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)(1024 >> 4) << 32;                // stride byte offset: next 8-row group
  d |= (uint64_t)1 << 46;                          // descriptor version (sm_100 family)
  d |= (uint64_t)2 << 61;                          // swizzle mode: 128 B
  return d;
}
// instruction descriptor: kind::f16, A = B = bf16, D = f32, both K-major, M x N
__device__ __forceinline__ uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}
__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
      ::"r"(tmem_d), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* v) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ int find_instance(const int* tstart, int n, int b) {
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (__ldg(tstart + mid) <= b) lo = mid; else hi = mid - 1;
  }
  return lo;
}
__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}
// 8 consecutive channels of an operand as fp32 (dt: bf16 or fp32; 16-byte aligned)
__device__ __forceinline__ void load8(const void* base, int dt, int64_t idx, float* v) {
  if (dt == DT_BF16) {
    const uint4 u = __ldg(reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(base) + idx));
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(h[i]);
      v[2 * i] = f.x;
      v[2 * i + 1] = f.y;
    }
  } else {
    const float4* p = reinterpret_cast<const float4*>(reinterpret_cast<const float*>(base) + idx);
    const float4 a = __ldg(p), b = __ldg(p + 1);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  }
}

struct TcShared {
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t accum;
  uint32_t tmem;
  int abort_flag;
  float red[4][256][2];
};

}  // namespace

// ---------------------------------------------------------------------------
// forward: Y[m][n] = sum_k act(X)[pix(m,k)] * W[n][k]  (+ res), BN partials
__global__ void __launch_bounds__(kThreads, 1) k_conv_fwd_tc(const ConvDesc* __restrict__ tab,
                                                             const int* __restrict__ tstart, int ninst,
                                                             int bnmax, int32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* const gbase = smem_raw + (base - raw);
  const int inst = find_instance(tstart, ninst, blockIdx.x);
  const ConvDesc& d = tab[inst];
  const int t = blockIdx.x - tstart[inst];
  const int tm = t % d.mtiles, tn = t / d.mtiles;
  const int BN = d.ntiles == 1 ? ((d.K + 15) & ~15) : 256;
  const int n0 = tn * 256;
  const int stage_bytes = kABytes + bnmax * 128;  // A + the launch's largest B tile
  TcShared& sh = *reinterpret_cast<TcShared*>(gbase + kStages * stage_bytes);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int M = d.B * d.P * d.Q;
  const int Kt = d.R * d.S * d.C;
  const int nkt = (Kt + kBK - 1) / kBK;
  const int m0 = tm * kBM;
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
  if (warp == 4) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&sh.tmem)),
                 "r"(ncols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sh.tmem;
  volatile int* abort_flag = &sh.abort_flag;

  if (warp < 4) {
    // ------------------------------------------------ producers
    const int cc = threadIdx.x & 7;        // 16-byte chunk within the 128-byte row
    const int rg = threadIdx.x >> 3;       // rows rg + 16 i
    int pn[8], ph[8], pw[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int m = m0 + rg + 16 * i;
      if (m < M) {
        const int q = m % d.Q, tmp = m / d.Q;
        pw[i] = q * d.stride - d.pad;
        ph[i] = (tmp % d.P) * d.stride - d.pad;
        pn[i] = tmp / d.P;
      } else {
        pn[i] = -1; ph[i] = 0; pw[i] = 0;
      }
    }
    bool ok = true;
    for (int kt = 0; kt < nkt && ok; ++kt) {
      const int s = kt % kStages;
      const uint32_t par = ((kt / kStages) & 1) ^ 1;
      if (!mbar_wait(smem_u32(&sh.empty[s]), par, abort_flag)) { ok = false; break; }
      uint8_t* A = gbase + s * stage_bytes;
      uint8_t* Bt = A + kABytes;
      const int k = kt * kBK + cc * 8;
      // A: im2col rows
      int c0 = 0, r_ = 0, s_ = 0;
      const bool kin = k < Kt;
      if (kin) {
        c0 = k % d.C;
        const int rs = k / d.C;
        s_ = rs % d.S;
        r_ = rs / d.S;
      }
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
            out.x = pack_bf16(v[0], v[1]);
            out.y = pack_bf16(v[2], v[3]);
            out.z = pack_bf16(v[4], v[5]);
            out.w = pack_bf16(v[6], v[7]);
          }
        }
        *reinterpret_cast<uint4*>(A + row * 128 + ((cc ^ (row & 7)) << 4)) = out;
      }
      // B: weight rows W[n0 + n][k .. k+7]
      for (int idx = threadIdx.x; idx < BN * 8; idx += 128) {
        const int n = idx >> 3, ch = idx & 7;
        const int kk = kt * kBK + ch * 8;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (n0 + n < d.K && kk < Kt)
          v = __ldg(reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(d.w) +
                                                   (int64_t)(n0 + n) * Kt + kk));
        *reinterpret_cast<uint4*>(Bt + n * 128 + ((ch ^ (n & 7)) << 4)) = v;
      }
      fence_proxy_async();
      mbar_arrive(smem_u32(&sh.full[s]));
    }
    if (!ok) {
      sh.abort_flag = 1;
      atomicExch(status, 3);
    }
    // ------------------------------------------------ epilogue
    bool got = ok && mbar_wait(smem_u32(&sh.accum), 0, abort_flag);
    if (!got && ok) { sh.abort_flag = 1; atomicExch(status, 3); }
    got = __all_sync(0xffffffffu, got);  // tcgen05.ld is warp-collective
    tc_fence_after();
    const int row = warp * 32 + lane;
    const int m = m0 + row;
    const bool mvalid = m < M;
    const uint32_t tbase = tmem + ((uint32_t)(warp * 32) << 16);
    for (int j0 = 0; j0 < BN; j0 += 16) {
      float v[16];
      if (got) tmem_ld16(tbase + j0, v);
      else
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = 0.f;
      const int nbase = n0 + j0;
      float s1[16], s2[16];
      if (mvalid && got) {
        const int64_t o = (int64_t)m * d.K + nbase;
        const bool full = nbase + 16 <= d.K;
        if (d.res) {
          if (full && (d.K % 8) == 0) {
            float r8[8];
            load8(d.res, d.res_dt, o, r8);
#pragma unroll
            for (int i = 0; i < 8; ++i) v[i] += r8[i];
            load8(d.res, d.res_dt, o + 8, r8);
#pragma unroll
            for (int i = 0; i < 8; ++i) v[8 + i] += r8[i];
          } else {
            for (int i = 0; i < 16; ++i)
              if (nbase + i < d.K)
                v[i] += d.res_dt == DT_F32 ? reinterpret_cast<const float*>(d.res)[o + i]
                                           : __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(d.res)[o + i]);
          }
        }
        if (d.y_dt == DT_BF16) {
#pragma unroll
          for (int i = 0; i < 16; ++i) v[i] = __bfloat162float(__float2bfloat16_rn(v[i]));
        }
        if (full && (d.K % 8) == 0) {
          if (d.y_dt == DT_BF16) {
            uint4 a, b;
            a.x = pack_bf16(v[0], v[1]); a.y = pack_bf16(v[2], v[3]); a.z = pack_bf16(v[4], v[5]); a.w = pack_bf16(v[6], v[7]);
            b.x = pack_bf16(v[8], v[9]); b.y = pack_bf16(v[10], v[11]); b.z = pack_bf16(v[12], v[13]); b.w = pack_bf16(v[14], v[15]);
            uint4* p = reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(d.y) + o);
            p[0] = a;
            p[1] = b;
          } else {
            float4* p = reinterpret_cast<float4*>(reinterpret_cast<float*>(d.y) + o);
            p[0] = make_float4(v[0], v[1], v[2], v[3]);
            p[1] = make_float4(v[4], v[5], v[6], v[7]);
            p[2] = make_float4(v[8], v[9], v[10], v[11]);
            p[3] = make_float4(v[12], v[13], v[14], v[15]);
          }
        } else {
          for (int i = 0; i < 16; ++i) {
            if (nbase + i >= d.K) break;
            if (d.y_dt == DT_BF16) reinterpret_cast<__nv_bfloat16*>(d.y)[o + i] = __float2bfloat16_rn(v[i]);
            else reinterpret_cast<float*>(d.y)[o + i] = v[i];
          }
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) { s1[i] = v[i]; s2[i] = v[i] * v[i]; }
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
    }
    if (d.stats) {
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
    // ------------------------------------------------ MMA issuer
    const uint32_t idesc = idesc_bf16(kBM, BN);
    bool ok = true;
    for (int kt = 0; kt < nkt; ++kt) {
      const int s = kt % kStages;
      if (!mbar_wait(smem_u32(&sh.full[s]), (kt / kStages) & 1, abort_flag)) { ok = false; break; }
      tc_fence_after();
      const uint32_t a_addr = base + s * stage_bytes;
      const uint32_t b_addr = a_addr + kABytes;
      const int ksub = min(4, (Kt - kt * kBK + 15) / 16);
      for (int kk = 0; kk < ksub; ++kk)
        mma_bf16(tmem, sw128_desc(a_addr + kk * 32), sw128_desc(b_addr + kk * 32), idesc, (kt | kk) ? 1u : 0u);
      mma_commit(smem_u32(&sh.empty[s]));
    }
    if (ok) {
      mma_commit(smem_u32(&sh.accum));
    } else {
      sh.abort_flag = 1;
      atomicExch(status, 3);
      // drain: the last committed stage barrier completes once all issued MMAs have
      mma_commit(smem_u32(&sh.accum));
      mbar_wait_drain(smem_u32(&sh.accum), 0);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 4) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(ncols));
  }
}

size_t conv_tc_smem_bytes(int bnmax) { return 1024 + kStages * (kABytes + (size_t)bnmax * 128) + sizeof(TcShared); }

cudaError_t launch_conv_fwd_tc(const ConvDesc* tab, const int* tstart, int n, int total, int bnmax, int32_t* status,
                               cudaStream_t st) {
  if (total <= 0) return cudaSuccess;
  if (bnmax < 16 || bnmax > 256 || (bnmax & 15)) return cudaErrorInvalidValue;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_conv_fwd_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)conv_tc_smem_bytes(256));
    if (e != cudaSuccess) return e;
    attr = true;
  }
  k_conv_fwd_tc<<<total, kThreads, conv_tc_smem_bytes(bnmax), st>>>(tab, tstart, n, bnmax, status);
  return cudaGetLastError();
}

}  // namespace pnn
