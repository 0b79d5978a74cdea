// Inline-PTX building blocks for the sm_103a tensor-core kernels: mbarriers
// with bounded waits, async-proxy fences, TMEM allocation, tcgen05.mma
// (kind::f16, bf16 operands, fp32 accumulator), tcgen05.commit and
// tcgen05.ld, plus shared-memory matrix descriptors for the 128-byte
// swizzled K-major layout.
#pragma once
#include <cuda_bf16.h>
#include <stdint.h>

namespace pnn {
namespace tc {

constexpr unsigned long long kWaitNs = 2000000000ull;  // 2 s budget per wait

// Debug builds (-DPNN_DEBUG_CHECKS) verify the alignment of every vector
// global access; the first violation is recorded as (line << 40 | address low
// 40 bits) in g_dbg and the access is skipped.  Release builds compile the
// checks away.
#ifdef PNN_DEBUG_CHECKS
__device__ unsigned long long g_dbg;
__device__ __forceinline__ bool dbg_ok(const void* p, unsigned a, int line) {
  const unsigned long long u = reinterpret_cast<unsigned long long>(p);
  if ((u & (a - 1)) == 0) return true;
  atomicCAS(&g_dbg, 0ull, ((unsigned long long)line << 40) | (u & 0xFFFFFFFFFFull));
  return false;
}
#define PNN_ALIGNED(p, a) ::pnn::tc::dbg_ok((p), (a), __LINE__)
#else
#define PNN_ALIGNED(p, a) true
#endif

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
// A waiting thread may be suspended for up to kSuspendNs inside one try_wait
// (it resumes as soon as the phase completes), so waiting warps leave the
// issue slots to the working ones.
#ifndef PNN_SUSPEND_NS
#define PNN_SUSPEND_NS 20000
#endif
constexpr uint32_t kSuspendNs = PNN_SUSPEND_NS;
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  if (kSuspendNs > 0) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity), "r"(kSuspendNs)
        : "memory");
  } else {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
  }
  return ok != 0;
}
// bounded wait: false after limit_ns or when another thread of the CTA aborted
__device__ __forceinline__ bool mbar_wait_for(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                              unsigned long long limit_ns) {
  if (mbar_try(bar, parity)) return true;
  const unsigned long long t0 = gtimer();
  while (true) {
    if (mbar_try(bar, parity)) return true;
    if (*abort_flag) return false;
    if (gtimer() - t0 > limit_ns) return false;
  }
}
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  return mbar_wait_for(bar, parity, abort_flag, kWaitNs);
}
// time-bounded wait that ignores the abort flag (drains committed MMAs)
__device__ __forceinline__ bool mbar_wait_drain(uint32_t bar, uint32_t parity) {
  const unsigned long long t0 = gtimer();
  while (!mbar_try(bar, parity))
    if (gtimer() - t0 > kWaitNs) return false;
  return true;
}
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tmem_alloc(uint32_t slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(slot), "r"(ncols));
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols));
}
// shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups 1024 B apart
__device__ __forceinline__ uint64_t sw128_desc(uint32_t addr) {
  uint64_t d = 0;
  d |= (uint64_t)((addr & 0x3FFFF) >> 4);  // start address
  d |= (uint64_t)1 << 16;                  // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)(1024 >> 4) << 32;        // stride byte offset: next 8-row group
  d |= (uint64_t)1 << 46;                  // descriptor version (sm_100 family)
  d |= (uint64_t)2 << 61;                  // swizzle mode: 128 B
  return d;
}
// shared-memory matrix descriptor: K-major, no swizzle.  Core matrices of 8
// rows x 16 bytes (rows 16 bytes apart, 128 contiguous bytes); lbo = bytes
// between core matrices adjacent in K, sbo = bytes between adjacent 8-row
// groups.  The start needs only 16-byte alignment, so a window that starts
// at any row of a row-contiguous plane is a valid operand.
__device__ __forceinline__ uint64_t nosw_desc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((addr & 0x3FFFF) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFF) << 32;
  d |= (uint64_t)1 << 46;                  // descriptor version (sm_100 family); swizzle mode 0: none
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
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
// 32 TMEM lanes x 16 fp32 columns -> 16 registers per thread
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

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}
__device__ __forceinline__ uint4 pack8(const float* v) {
  return make_uint4(pack_bf16(v[0], v[1]), pack_bf16(v[2], v[3]), pack_bf16(v[4], v[5]), pack_bf16(v[6], v[7]));
}
// 8 consecutive elements as fp32 (dt 1 = bf16, 0 = fp32; 16-byte aligned address)
__device__ __forceinline__ void load8(const void* base, int dt, int64_t idx, float* v) {
  if (dt == 1) {
    const uint4* q = reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(base) + idx);
    if (!PNN_ALIGNED(q, 16)) {
      for (int i = 0; i < 8; ++i) v[i] = 0.f;
      return;
    }
    const uint4 u = __ldg(q);
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(h[i]);
      v[2 * i] = f.x;
      v[2 * i + 1] = f.y;
    }
  } else {
    const float4* p = reinterpret_cast<const float4*>(reinterpret_cast<const float*>(base) + idx);
    if (!PNN_ALIGNED(p, 16)) {
      for (int i = 0; i < 8; ++i) v[i] = 0.f;
      return;
    }
    const float4 a = __ldg(p), b = __ldg(p + 1);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  }
}
// 8x8 transpose of bf16: in[p] holds 8 elements e[p][0..7]; out[c] = e[0..7][c]
__device__ __forceinline__ void transpose8(const uint4* in, uint4* out) {
  const uint32_t* w = reinterpret_cast<const uint32_t*>(in);  // w[p*4 + c/2], half c%2
  uint32_t* o = reinterpret_cast<uint32_t*>(out);              // o[c*4 + p/2], half p%2
#pragma unroll
  for (int c = 0; c < 8; ++c)
#pragma unroll
    for (int p = 0; p < 8; p += 2) {
      const uint32_t a = w[p * 4 + c / 2], b = w[(p + 1) * 4 + c / 2];
      o[c * 4 + p / 2] = __byte_perm(a, b, (c & 1) ? 0x7632 : 0x5410);
    }
}
// 16-byte global -> shared copy that does not block the issuing thread
// (L2-cached); n_src < 16 fills the rest of the 16 bytes with zeros (0: all
// zeros, nothing is read).  cp_async_wait_all() waits for this thread's copies.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int n_src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n_src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }
// arrive on the mbarrier and add `bytes` to the transaction count its current
// phase waits for (the TMA copies that complete_tx on it)
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
// 2-D tiled TMA load of one box at element coordinates (x inner, y outer) of
// the tensor map (global memory, 128-byte aligned) into shared memory; the
// copy completes `bytes of the box` on the mbarrier.  x * element size must be
// a multiple of 16 bytes; y may lie outside the tensor (zero fill).
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void* tmap, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(dst), "l"(tmap), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
// 2-D tiled TMA store of one box from shared memory to element coordinates
// (x inner, y outer) of the tensor map; parts of the box outside the tensor
// are not written.  x * element size must be a multiple of 16 bytes and both
// coordinates non-negative.  Completion is tracked per thread by bulk groups.
__device__ __forceinline__ void tma_store_2d(const void* tmap, int x, int y, uint32_t src) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(tmap), "r"(x),
               "r"(y), "r"(src)
               : "memory");
}
// the same box added element-wise (fp32) into global memory (done in L2)
__device__ __forceinline__ void tma_reduce_add_2d(const void* tmap, int x, int y, uint32_t src) {
  asm volatile("cp.reduce.async.bulk.tensor.2d.global.shared::cta.add.tile.bulk_group [%0, {%1, %2}], [%3];" ::"l"(tmap),
               "r"(x), "r"(y), "r"(src)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// wait until at most N of this thread's bulk groups still read shared memory
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
// wait until all of this thread's bulk groups are complete
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// byte offset of 16-byte chunk `ch` of row `row` in the 128-byte-swizzled K-major layout
__device__ __forceinline__ uint32_t swz(int row, int ch) { return (uint32_t)(row * 128 + ((ch ^ (row & 7)) << 4)); }

}  // namespace tc
}  // namespace pnn
