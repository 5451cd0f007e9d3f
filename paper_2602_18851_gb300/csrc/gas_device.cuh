// Device-side helpers shared by the library's kernels (sm_103a).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "gas_internal.h"

namespace gas {

// ---------------------------------------------------------------------------------
// bf16 <-> fp32 (bf16 is the top half of an fp32: widening is exact)
// ---------------------------------------------------------------------------------
__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ void unpack8(const uint4& q, float (&f)[8]) {
  f[0] = bf16lo(q.x); f[1] = bf16hi(q.x);
  f[2] = bf16lo(q.y); f[3] = bf16hi(q.y);
  f[4] = bf16lo(q.z); f[5] = bf16hi(q.z);
  f[6] = bf16lo(q.w); f[7] = bf16hi(q.w);
}

// Eight binary16 values (one 16-byte load) widened exactly to fp32.
__device__ __forceinline__ void unpack8_f16(const uint4& q, float (&f)[8]) {
  const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 v = __half22float2(*reinterpret_cast<const __half2*>(&w[i]));
    f[2 * i] = v.x;
    f[2 * i + 1] = v.y;
  }
}

// Eight weights of the handle's format (bf16, or binary16 when F16).
template <bool F16>
__device__ __forceinline__ void unpack8w(const uint4& q, float (&f)[8]) {
  if (F16) unpack8_f16(q, f);
  else unpack8(q, f);
}

// Weight element types of the CUDA-core kernels: bf16, binary16, fp32.
enum WeightType : int { kWBf16 = 0, kWF16 = 1, kWF32 = 2 };

// Eight consecutive weights (16 bytes of 16-bit values, 32 bytes of fp32) as loaded.
template <int WT>
struct W8 {
  uint4 q[WT == kWF32 ? 2 : 1];
};

// Streaming (evict-first) load of the eight weights at element offset `off` of `base`.
template <int WT>
__device__ __forceinline__ W8<WT> load_w8(const void* base, long long off) {
  W8<WT> w;
  if (WT == kWF32) {
    const uint4* p = reinterpret_cast<const uint4*>(static_cast<const float*>(base) + off);
    w.q[0] = __ldcs(p);
    w.q[1] = __ldcs(p + 1);
  } else {
    w.q[0] = __ldcs(reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(base) + off));
  }
  return w;
}

template <int WT>
__device__ __forceinline__ W8<WT> zero_w8() {
  W8<WT> w;
#pragma unroll
  for (int i = 0; i < (WT == kWF32 ? 2 : 1); ++i) w.q[i] = make_uint4(0, 0, 0, 0);
  return w;
}

template <int WT>
__device__ __forceinline__ void unpack_w8(const W8<WT>& w, float (&f)[8]) {
  if (WT == kWBf16) {
    unpack8(w.q[0], f);
  } else if (WT == kWF16) {
    unpack8_f16(w.q[0], f);
  } else {
    const uint32_t b[8] = {w.q[0].x, w.q[0].y, w.q[0].z, w.q[0].w, w.q[1].x, w.q[1].y, w.q[1].z, w.q[1].w};
#pragma unroll
    for (int i = 0; i < 8; ++i) f[i] = __uint_as_float(b[i]);
  }
}

// Round-to-nearest-even fp32 -> bf16 bits.
__device__ __forceinline__ uint32_t f32_to_bf16_bits(float x) {
  return static_cast<uint32_t>(__bfloat16_as_ushort(__float2bfloat16_rn(x)));
}

// ---------------------------------------------------------------------------------
// Reductions
// ---------------------------------------------------------------------------------
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, off);
  return v;
}

// Each lane holds R partial values (R a power of two, 2..32).  On return v[0] holds
// the sum over all 32 lanes of value number `idx` (returned), with log2(R) exchange
// steps that halve the live values plus the remaining butterfly steps:
// 16 shuffles for R = 16 instead of 5 * R.
template <int R>
__device__ __forceinline__ float warp_transpose_reduce(float (&v)[R], int lane, int& idx) {
  int base = 0;
#pragma unroll
  for (int n = R, off = 16; n > 1; n >>= 1, off >>= 1) {
    const int h = n >> 1;
    const bool up = (lane & off) != 0;
#pragma unroll
    for (int k = 0; k < h; ++k) {
      const float send = up ? v[k] : v[k + h];
      const float keep = up ? v[k + h] : v[k];
      v[k] = keep + __shfl_xor_sync(0xFFFFFFFFu, send, off);
    }
    if (up) base += h;
  }
#pragma unroll
  for (int off = 16 / R; off >= 1; off >>= 1) v[0] += __shfl_xor_sync(0xFFFFFFFFu, v[0], off);
  idx = base;
  return v[0];
}

// Lanes that hold a distinct result after warp_transpose_reduce<R>.
template <int R>
__device__ __forceinline__ bool transpose_reduce_writer(int lane) {
  return (lane & (32 / R - 1)) == 0;
}

__device__ __forceinline__ float safe_inv_sqrt(float s2) {
  // 1/sqrt(s2) with the zero guard of the method's reading (0 for a zero norm).
  return s2 > 0.0f ? rsqrtf(s2) : (s2 == 0.0f ? 0.0f : __int_as_float(0x7FC00000));
}

__device__ __forceinline__ void set_status(unsigned* status, unsigned bits) {
  if (status) atomicOr(status, bits);
}

// Max of non-negative floats (or NaN) through their bit patterns; NaN dominates.
__device__ __forceinline__ void atomic_max_nonneg(float* dst, float v) {
  const float w = (v == 0.0f) ? 0.0f : v;  // no -0.0
  atomicMax(reinterpret_cast<unsigned*>(dst), __float_as_uint(w));
}

// ---------------------------------------------------------------------------------
// Shared-memory addresses, mbarriers (bounded waits), TMA, tcgen05
// ---------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ uint32_t mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok;
}

// Wait for the phase with parity `parity` of an mbarrier to complete, for at most
// kWaitLimitNs.  Gives up early when another role of the CTA raised *abort.
// Returns false (and flags the device status word) on timeout or abort.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort,
                                          unsigned* status) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t spin = 1;; ++spin) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((spin & 255u) == 0u) {
      if (*abort) return false;
      if (global_timer_ns() - t0 > kWaitLimitNs) {
        *abort = 1;
        set_status(status, GAS_DEV_WAIT_TIMEOUT);
        return false;
      }
    }
  }
}

__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap* m) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(m)) : "memory");
}

// 2D tiled TMA load of box {x .. x+bx, y .. y+by} into shared memory; completion is
// signalled on `bar` as transaction bytes.  x * sizeof(elem) must be a multiple of 16.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                            int x, int y, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y), "l"(policy)
      : "memory");
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                            int x, int y, int z, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%3, %4, %5}], [%2], %6;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y), "r"(z), "l"(policy)
      : "memory");
}

// --- tcgen05 (5th-generation tensor core, accumulators in tensor memory) -----------
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (bf16 inputs, fp32 accumulate), one CTA.
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                          uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on `bar` when every tcgen05 op issued so far by this thread has completed.
__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   bar)
               : "memory");
}

// 32 lanes x 16 consecutive 32-bit columns: thread t of the warp receives row
// (lane_base + t), columns col .. col+15.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor for a K-major operand stored with the 128-byte
// swizzle that a TMA box of 64 bf16 columns produces: rows of 128 B, 8-row groups of
// 1024 B (stride byte offset), descriptor version 1 (sm_100 family), layout
// SWIZZLE_128B.  Advancing K by 16 elements inside the 128-byte row adds 32 B to the
// start address (the hardware applies the swizzle on absolute address bits, so the
// tile base must be 1024-byte aligned).
__device__ __forceinline__ uint64_t desc_kmajor_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>(1u) << 16;           // leading byte offset (unused here)
  d |= static_cast<uint64_t>(1024u >> 4) << 32;   // stride byte offset
  d |= static_cast<uint64_t>(1u) << 46;           // version
  d |= static_cast<uint64_t>(2u) << 61;           // SWIZZLE_128B
  return d;
}

// Descriptor for an MN-major operand in the 128-byte-swizzled layout a TMA box of 64
// bf16 columns x R rows produces when the 64 contiguous columns are the M/N index
// and the rows are K: one 64-element swizzle atom across M/N, 8-row K groups 1024 B
// apart (stride byte offset).  Advancing K by 16 adds 2048 B to the start address.
__device__ __forceinline__ uint64_t desc_mnmajor_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>(1u) << 16;           // leading byte offset (one atom: unused)
  d |= static_cast<uint64_t>(1024u >> 4) << 32;   // stride byte offset: next 8 K rows
  d |= static_cast<uint64_t>(1u) << 46;
  d |= static_cast<uint64_t>(2u) << 61;
  return d;
}

// As desc_mnmajor_sw128 for an operand two swizzle atoms (128 elements) wide along
// M/N: the second 64-element atom starts `atom_stride` bytes after the first (leading
// byte offset), e.g. the second of two TMA boxes placed back to back.
__device__ __forceinline__ uint64_t desc_mnmajor_sw128_2atoms(uint32_t saddr, uint32_t atom_stride) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>((atom_stride >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>(1024u >> 4) << 32;
  d |= static_cast<uint64_t>(1u) << 46;
  d |= static_cast<uint64_t>(2u) << 61;
  return d;
}

// Generic-proxy shared-memory writes become visible to the tensor core (async proxy).
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, both K-major.
// x as a hi + lo pair of 16-bit operands of the weights' format (bf16, or binary16):
// hi = RN(x), lo = RN(x - hi).
__device__ __forceinline__ void split_hilo(float x, bool f16, uint32_t& hb, uint32_t& lb) {
  if (f16) {
    const __half h = __float2half_rn(x);
    hb = __half_as_ushort(h);
    lb = __half_as_ushort(__float2half_rn(x - __half2float(h)));
  } else {
    hb = f32_to_bf16_bits(x);
    lb = f32_to_bf16_bits(x - __uint_as_float(hb << 16));
  }
}

__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
  return (1u << 4)                                 // D format: f32
         | (1u << 7)                               // A format: bf16
         | (1u << 10)                              // B format: bf16
         | (static_cast<uint32_t>(N >> 3) << 17)   // N / 8
         | (static_cast<uint32_t>(M >> 4) << 24);  // M / 16
}

// kind::f16 descriptor for bf16 (f16 == false) or binary16 operands (A and B alike).
__host__ __device__ constexpr uint32_t idesc_f32acc(int M, int N, bool f16) {
  return f16 ? (idesc_bf16_f32(M, N) & ~((1u << 7) | (1u << 10))) : idesc_bf16_f32(M, N);
}

// As idesc_bf16_f32 with A MN-major ("transpose A").
__host__ __device__ constexpr uint32_t idesc_bf16_f32_amn(int M, int N) {
  return idesc_bf16_f32(M, N) | (1u << 15);
}

// As idesc_bf16_f32 with B MN-major ("transpose B").
__host__ __device__ constexpr uint32_t idesc_bf16_f32_bmn(int M, int N) {
  return idesc_bf16_f32(M, N) | (1u << 16);
}

// Programmatic dependent launch: a kernel launched with programmatic stream
// serialization may start once every CTA of the kernel before it has called
// griddep_launch_dependents (or exited); griddep_wait then blocks until that kernel has
// completed and its memory operations are visible.  Without the launch attribute the
// wait returns at once.
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// ---------------------------------------------------------------------------------
// Named barriers, flags, wide tensor-memory loads
// ---------------------------------------------------------------------------------
__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// Named barrier with an AND vote: every participating thread gets the AND of `v`.
__device__ __forceinline__ bool named_bar_and(int id, int nthreads, bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.and.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(v)), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release_u32(unsigned* p, unsigned v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Bounded wait for another CTA's key tile: true once *flag == epoch.
__device__ inline bool wait_flag(const unsigned* flag, unsigned epoch, volatile int* abort, unsigned* status) {
  const uint64_t t0 = global_timer_ns();
  for (;;) {
    if (ld_acquire_u32(flag) == epoch) return true;
    if (*abort) return false;
    if (global_timer_ns() - t0 > kWaitLimitNs) {
      *abort = 1;
      set_status(status, GAS_DEV_WAIT_TIMEOUT);
      return false;
    }
    __nanosleep(128);
  }
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]),
        "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]),
        "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

}  // namespace gas
