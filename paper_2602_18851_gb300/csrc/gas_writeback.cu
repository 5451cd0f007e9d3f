// Tensor-core write-back of the right singular vector estimates (Algorithm 2's final
// v = v'/||v'||, needed for the warm start of the next refresh, Section 4.1):
//
//   v_out[h] = B_g^T (y_h / ||v'_h||)   for every head h of KV group g,
//
// one more pass over every key block B_g (d_h x d bf16).  Per key tile (128 rows = one
// or two groups) and 64-column chunk c0.. of d it is one tcgen05 MMA chain
//   D[n][c] = sum_i Y[n][i] * B[i][c],   M = 128 (n), N = 64 (c), K = 128 (i),
// with A = Y split into bf16 hi and lo rows (about 16 bits of mantissa, K-major, staged
// in shared memory by the epilogue warps) and B = the TMA box of the weight tile read
// MN-major (its 64 contiguous columns are the N index).  Row layout of Y: head j of
// group gi of the tile is number u = gi*G + j; it goes to TMEM lane quarter u % 4 (so
// all four epilogue warps drain D), slot m = u / 4: hi part in row 32*(u%4) + m, lo part
// in row 32*(u%4) + 16 + m, non-zero only in the group's own K range.  The epilogue adds
// the hi and lo rows with one shuffle inside a warp.  Group size <= 16.

#include "gas_device.cuh"

namespace gas {

namespace {

constexpr int kWbThreads = 192;            // warp 0 TMA, warp 1 MMA, warps 2-5 stage Y / drain D
constexpr int kWbCols = 1024;              // columns of d per work item
constexpr int kWbStages = 9;
constexpr int kWbSlots = 4;                // tensor-memory accumulators of 64 columns
constexpr uint32_t kBox = 128u * 64u * 2u; // 64 columns x 128 rows bf16
constexpr uint32_t kYBytes = 2u * 16384u;  // 128 rows x 128 K bf16 as two 64-wide K atoms
constexpr size_t kWbSmem = 2 * kYBytes + kWbStages * kBox + 4096;

struct WbItem {
  int layer, tile, c0, nchunks;
};

__device__ __forceinline__ WbItem decode_item(const Shape& s, int t) {
  const int ncb = (s.d + kWbCols - 1) / kWbCols;
  WbItem w;
  w.layer = t / (s.tiles_k * ncb);
  const int rem = t - w.layer * s.tiles_k * ncb;
  w.tile = rem / ncb;
  w.c0 = (rem - w.tile * ncb) * kWbCols;
  const int ncols = min(kWbCols, s.d - w.c0);
  w.nchunks = (ncols + 63) / 64;
  return w;
}

template <int DH>
__global__ void __launch_bounds__(kWbThreads, 1) writeback_kernel(const __grid_constant__ WbArgs a) {
  constexpr int S = kWbStages;
  constexpr int GPT = 128 / DH;  // groups per key tile
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* ybuf_s = smem;                    // [2][kYBytes]
  uint8_t* ring = smem + 2 * kYBytes;        // [S][kBox]
  uint64_t* bars = reinterpret_cast<uint64_t*>(ring + S * kBox);
  uint64_t* full = bars;
  uint64_t* empty = full + S;
  uint64_t* yfull = empty + S;
  uint64_t* yempty = yfull + 2;
  uint64_t* dfull = yempty + 2;
  uint64_t* dempty = dfull + kWbSlots;
  uint64_t* done = dempty + kWbSlots;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int no_abort_flag = 0;

  const Shape& s = a.s;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&yfull[i]), 128);
      mbar_init(smem_u32(&yempty[i]), 1);
    }
    for (int i = 0; i < kWbSlots; ++i) {
      mbar_init(smem_u32(&dfull[i]), 1);
      mbar_init(smem_u32(&dempty[i]), 128);
    }
    mbar_init(smem_u32(done), 1);
    *abort = 0;
    fence_mbar_init();
  }
  // Rows and K ranges of Y that no head uses stay zero for the whole launch.
  for (uint32_t o = threadIdx.x * 16u; o < 2u * kYBytes; o += kWbThreads * 16u)
    *reinterpret_cast<uint4*>(ybuf_s + o) = make_uint4(0, 0, 0, 0);
  fence_proxy_async_smem();
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int ncb = (s.d + kWbCols - 1) / kWbCols;
  const int T = s.L * s.tiles_k * ncb;

  if (warp == 0) {
    if (lane == 0) {
      const uint64_t pol = l2_policy_evict_first();
      uint32_t issued = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < T && ok; t += gridDim.x) {
        const WbItem w = decode_item(s, t);
        for (int j = 0; j < w.nchunks; ++j) {
          const uint32_t st = issued % S, ph = (issued / S) & 1u;
          if (!mbar_wait(smem_u32(&empty[st]), ph ^ 1u, abort, a.status)) { ok = false; break; }
          const uint32_t fb = smem_u32(&full[st]);
          mbar_arrive_expect_tx(fb, kBox);
          tma_load_2d(smem_u32(ring + st * kBox), &a.maps_k[w.layer], fb, w.c0 + 64 * j, w.tile * 128, pol);
          ++issued;
        }
      }
      const uint32_t first = issued > static_cast<uint32_t>(S) ? issued - S : 0u;
      for (uint32_t i = first; i < issued; ++i)
        mbar_wait(smem_u32(&full[i % S]), (i / S) & 1u, &no_abort_flag, a.status);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32_bmn(128, 64);
      uint32_t consumed = 0, cc = 0, it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < T && ok; t += gridDim.x, ++it) {
        const WbItem w = decode_item(s, t);
        const uint32_t yb = it & 1u;
        if (!mbar_wait(smem_u32(&yfull[yb]), (it >> 1) & 1u, abort, a.status)) break;
        tc_fence_after();
        const uint32_t ybase = smem_u32(ybuf_s + yb * kYBytes);
        for (int j = 0; j < w.nchunks; ++j, ++cc) {
          const uint32_t slot = cc % kWbSlots;
          if (!mbar_wait(smem_u32(&dempty[slot]), ((cc / kWbSlots) & 1u) ^ 1u, abort, a.status)) { ok = false; break; }
          const uint32_t st = consumed % S, ph = (consumed / S) & 1u;
          if (!mbar_wait(smem_u32(&full[st]), ph, abort, a.status)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sx = smem_u32(ring + st * kBox);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint64_t ad = desc_kmajor_sw128(ybase + (kk >> 2) * 16384u + (kk & 3) * 32u);
            const uint64_t bd = desc_mnmajor_sw128(sx + kk * 2048u);
            umma_bf16(tmem + slot * 64u, ad, bd, idesc, kk > 0 ? 1u : 0u);
          }
          umma_commit(smem_u32(&empty[st]));
          umma_commit(smem_u32(&dfull[slot]));
          ++consumed;
        }
        if (!ok) break;
        umma_commit(smem_u32(&yempty[yb]));
      }
      umma_commit(smem_u32(done));
      mbar_wait(smem_u32(done), 0u, &no_abort_flag, a.status);
    }
  } else {
    const int ethr = threadIdx.x - 64;
    const int q = warp & 3;
    const int G = s.G;
    const int units = GPT * G * (DH / 8);
    uint32_t staged = 0;
    // Stage Y (hi/lo bf16, swizzled K-major) of item t into buffer staged & 1.
    auto stage = [&](int t) -> bool {
      const WbItem w = decode_item(s, t);
      const uint32_t yb = staged & 1u;
      const bool ok = mbar_wait(smem_u32(&yempty[yb]), ((staged >> 1) & 1u) ^ 1u, abort, a.status);
      if (ok) {
        uint8_t* ybase = ybuf_s + yb * kYBytes;
        for (int u = ethr; u < units; u += 128) {
          const int gi = u / (G * (DH / 8));
          const int rem = u - gi * G * (DH / 8);
          const int j = rem / (DH / 8);
          const int i0 = (rem - j * (DH / 8)) * 8;
          const int g = w.tile * GPT + gi;
          float v[8];
          if (g < s.nkv) {
            const float* src = a.ybuf + (static_cast<size_t>(w.layer) * s.nq + g * G + j) * DH + i0;
            const float4 a0 = *reinterpret_cast<const float4*>(src);
            const float4 a1 = *reinterpret_cast<const float4*>(src + 4);
            v[0] = a0.x; v[1] = a0.y; v[2] = a0.z; v[3] = a0.w;
            v[4] = a1.x; v[5] = a1.y; v[6] = a1.z; v[7] = a1.w;
          } else {
#pragma unroll
            for (int e = 0; e < 8; ++e) v[e] = 0.0f;
          }
          uint32_t hb[8], lb[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            hb[e] = f32_to_bf16_bits(v[e]);
            lb[e] = f32_to_bf16_bits(v[e] - __uint_as_float(hb[e] << 16));
          }
          const int k = gi * DH + i0;                 // K index of the 8-element chunk
          const int region = k >> 6, chunk = (k & 63) >> 3;
          const int hu = gi * G + j;                  // head slot u -> quarter u%4, row u/4
          const int rhi = 32 * (hu & 3) + (hu >> 2), rlo = rhi + 16;
          uint8_t* base = ybase + region * 16384;
          *reinterpret_cast<uint4*>(base + rhi * 128 + ((chunk ^ (rhi & 7)) << 4)) =
              make_uint4(hb[0] | (hb[1] << 16), hb[2] | (hb[3] << 16), hb[4] | (hb[5] << 16), hb[6] | (hb[7] << 16));
          *reinterpret_cast<uint4*>(base + rlo * 128 + ((chunk ^ (rlo & 7)) << 4)) =
              make_uint4(lb[0] | (lb[1] << 16), lb[2] | (lb[3] << 16), lb[4] | (lb[5] << 16), lb[6] | (lb[7] << 16));
        }
        fence_proxy_async_smem();
      }
      mbar_arrive(smem_u32(&yfull[yb]));
      ++staged;
      return ok;
    };
    uint32_t cc = 0;
    bool ok = true;
    // Every stage() is followed by a vote so that all four warps leave together.
    if (blockIdx.x < T) ok = named_bar_and(5, 128, stage(blockIdx.x));
    for (int t = blockIdx.x; t < T && ok; t += gridDim.x) {
      if (t + static_cast<int>(gridDim.x) < T) ok = named_bar_and(5, 128, stage(t + gridDim.x));
      if (!ok) break;
      const WbItem w = decode_item(s, t);
      for (int j = 0; j < w.nchunks; ++j, ++cc) {
        const uint32_t slot = cc % kWbSlots;
        const bool got = mbar_wait(smem_u32(&dfull[slot]), (cc / kWbSlots) & 1u, abort, a.status);
        __syncwarp();
        if (!named_bar_and(4, 128, got)) { ok = false; break; }
        tc_fence_after();
        if (q < GPT * G) {  // this lane quarter holds at least one head
          uint32_t r0[32], r1[32];
          const uint32_t taddr = tmem + (static_cast<uint32_t>(q * 32) << 16) + slot * 64u;
          tmem_ld32(taddr, r0);
          tmem_ld32(taddr + 32u, r1);
          tmem_ld_wait();
          float o[64];
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            const float hi0 = __uint_as_float(r0[c]), hi1 = __uint_as_float(r1[c]);
            o[c] = hi0 + __shfl_down_sync(0xFFFFFFFFu, hi0, 16);
            o[32 + c] = hi1 + __shfl_down_sync(0xFFFFFFFFu, hi1, 16);
          }
          const int hu = 4 * lane + q;  // head slot held by this lane's hi row
          const int g = w.tile * GPT + hu / G;
          if (lane < 16 && hu < GPT * G && g < s.nkv) {
            const int col0 = w.c0 + 64 * j;
            float* dst = a.v_out + (static_cast<size_t>(w.layer) * s.nq + g * G + hu % G) * s.d + col0;
#pragma unroll
            for (int c = 0; c < 64; c += 4)
              if (col0 + c < s.d) *reinterpret_cast<float4*>(dst + c) = make_float4(o[c], o[c + 1], o[c + 2], o[c + 3]);
          }
        }
        tc_fence_before();
        mbar_arrive(smem_u32(&dempty[slot]));
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
}

template <int DH>
cudaError_t launch_wb_dh(const WbArgs& a, int num_sms, cudaStream_t st) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(writeback_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(kWbSmem));
    if (e != cudaSuccess) return e;
    configured = true;
  }
  const int ncb = (a.s.d + kWbCols - 1) / kWbCols;
  const int T = a.s.L * a.s.tiles_k * ncb;
  const int grid = T < num_sms ? T : num_sms;
  writeback_kernel<DH><<<grid, kWbThreads, kWbSmem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_writeback(const WbArgs& a, int num_sms, cudaStream_t st) {
  if (a.s.G > kWbMaxGroup) return cudaErrorInvalidValue;
  if (a.s.dh == 128) return launch_wb_dh<128>(a, num_sms, st);
  if (a.s.dh == 64) return launch_wb_dh<64>(a, num_sms, st);
  return cudaErrorInvalidValue;
}

}  // namespace gas
