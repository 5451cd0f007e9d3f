// Tensor-core write-back of the right singular vector estimates (Algorithm 2's final
// v = v'/||v'||, needed for the warm start of the next refresh, Section 4.1):
//
//   v_out[h] = B_g^T (y_h / ||v'_h||)   for every head h of KV group g,
//
// one more pass over every key block B_g (d_h x d bf16).  Per key tile (128 rows = one
// or two groups) and 128-column chunk c0.. of d it is one tcgen05 MMA chain
//   D[c][n] = sum_i B[i][c] * Y[n][i],   M = 128 (c), N = nz (n), K = 128 (i),
// with A = two TMA boxes of the weight tile read MN-major (their contiguous columns are
// the M index) and B = Y, the vectors split into bf16 hi and lo rows (about 16 bits of
// mantissa), K-major, staged in shared memory by the epilogue warps.  Row layout of Y:
// head j of group gi of the tile is slot u = gi*G + j; its hi part is row u, its lo
// part row nz/2 + u, non-zero only in the group's own K range.  Each epilogue thread
// owns one column c (a TMEM lane) and adds rows u and nz/2 + u for every head, so a
// warp writes 32 consecutive floats of each head's v_out row.

#include "gas_device.cuh"

namespace gas {

namespace {

constexpr int kWbThreads = 192;               // warp 0 TMA, warp 1 MMA, warps 2-5 stage Y / drain D
constexpr int kWbCols = 1024;                 // columns of d per work item
constexpr int kWbSlots = 4;                   // tensor-memory accumulators of nz columns
constexpr uint32_t kBox = 128u * 64u * 2u;    // 64 columns x 128 rows bf16
constexpr uint32_t kStage = 2 * kBox;         // 128 columns
constexpr int kWbSmemBudget = 232448;         // 227 KB opt-in dynamic shared memory

template <int NZ>
struct WbCfg {
  static constexpr uint32_t kYBytes = 2u * NZ * 128u;  // nz rows x 128 K as two 64-wide K atoms
  static constexpr int kStages =
      (kWbSmemBudget - 4096 - 2 * static_cast<int>(kYBytes)) / static_cast<int>(kStage) > 6
          ? 6
          : (kWbSmemBudget - 4096 - 2 * static_cast<int>(kYBytes)) / static_cast<int>(kStage);
  static constexpr size_t kSmem = 2 * kYBytes + kStages * kStage + 4096;
  static constexpr uint32_t kTmemCols = (kWbSlots * NZ < 32) ? 32 : kWbSlots * NZ;
  static_assert(kYBytes % 1024 == 0, "Y atoms must stay 1024-byte aligned");
  static_assert(kStages >= 3, "ring too shallow");
};

struct WbItem {
  int layer, tile, c0, nchunks;
};

// Items walk the layers from the last one down: the Gram launch read the key tiles of
// its last layers most recently (and keeps them in L2), so the first items hit L2.
__device__ __forceinline__ WbItem decode_item(const Shape& s, int t) {
  const int ncb = (s.d + kWbCols - 1) / kWbCols;
  WbItem w;
  const int lr = t / (s.tiles_k * ncb);
  w.layer = s.L - 1 - lr;
  const int rem = t - lr * s.tiles_k * ncb;
  w.tile = rem / ncb;
  w.c0 = (rem - w.tile * ncb) * kWbCols;
  const int ncols = min(kWbCols, s.d - w.c0);
  w.nchunks = (ncols + 127) / 128;
  return w;
}

// GENERIC: binary16 weights or the Conv1D layout, chosen at run time (folded away in the
// default bf16 nn.Linear instantiation).
template <int DH, int NZ, bool GENERIC>
__global__ void __launch_bounds__(kWbThreads, 1) writeback_kernel(const __grid_constant__ WbArgs a) {
  using Cfg = WbCfg<NZ>;
  constexpr int S = Cfg::kStages;
  constexpr int GPT = 128 / DH;  // groups per key tile
  constexpr uint32_t YB = Cfg::kYBytes;
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte alignment by pointer arithmetic on the shared array itself, so that the
  // compiler keeps every derived pointer in the shared address space.
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint8_t* ring = smem;                      // [S][kStage]
  uint8_t* ybuf_s = smem + S * kStage;       // [2][YB]
  uint64_t* bars = reinterpret_cast<uint64_t*>(ybuf_s + 2 * YB);
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
  const bool cols = GENERIC && s.cols != 0;
  const bool f16 = GENERIC && s.f16 != 0;
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
  for (uint32_t o = threadIdx.x * 16u; o < 2u * YB; o += kWbThreads * 16u)
    *reinterpret_cast<uint4*>(ybuf_s + o) = make_uint4(0, 0, 0, 0);
  // A d_h 80 / 96 head fills only the top d_h rows (K) of its box; the rest stay zero.
  const uint32_t wbox = cols ? kBox : static_cast<uint32_t>((128 / DH) * a.s.rows) * 128u;
  if (wbox < kBox)
    for (int st = 0; st < S; ++st)
      for (int b = 0; b < 2; ++b)
        for (uint32_t o = wbox + threadIdx.x * 16u; o < kBox; o += kWbThreads * 16u)
          *reinterpret_cast<uint4*>(ring + st * kStage + b * kBox + o) = make_uint4(0, 0, 0, 0);
  fence_proxy_async_smem();
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), Cfg::kTmemCols);
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
          // The first S stages go out at once (W^K does not depend on the previous kernel);
          // the bounded waits for stages to drain start after that kernel has completed.
          if (issued == static_cast<uint32_t>(S)) griddep_wait();
          if (!mbar_wait(smem_u32(&empty[st]), ph ^ 1u, abort, a.status)) { ok = false; break; }
          const uint32_t fb = smem_u32(&full[st]);
          const uint32_t dst = smem_u32(ring + st * kStage);
          mbar_arrive_expect_tx(fb, 2u * wbox);
          if (cols) {
            // Conv1D: box b holds rows (K) 64b.. of the tile for the 128 columns (M),
            // K-major, fetched as two 64-column halves of 64-row boxes
#pragma unroll
            for (int b = 0; b < 2; ++b)
#pragma unroll
              for (int hh = 0; hh < 2; ++hh)
                tma_load_2d(dst + b * kBox + hh * (kBox / 2), &a.maps_k[w.layer], fb, w.tile * 128 + 64 * b,
                            w.c0 + 128 * j + 64 * hh, pol);
          } else {
            tma_load_3d(dst, &a.maps_k[w.layer], fb, w.c0 + 128 * j, 0, w.tile * (128 / DH), pol);
            tma_load_3d(dst + kBox, &a.maps_k[w.layer], fb, w.c0 + 128 * j + 64, 0, w.tile * (128 / DH), pol);
          }
          ++issued;
        }
      }
      const uint32_t first = issued > static_cast<uint32_t>(S) ? issued - S : 0u;
      for (uint32_t i = first; i < issued; ++i)
        mbar_wait(smem_u32(&full[i % S]), (i / S) & 1u, &no_abort_flag, a.status);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // A (the weight tile) is MN-major in the nn.Linear layout, K-major in the Conv1D one
      const uint32_t idesc = idesc_f32acc(128, NZ, f16) | (cols ? 0u : (1u << 15));
      uint32_t consumed = 0, cc = 0, it = 0;
      bool ok = true;
      griddep_wait();  // its bounded waits start once the previous kernel has completed
      for (int t = blockIdx.x; t < T && ok; t += gridDim.x, ++it) {
        const WbItem w = decode_item(s, t);
        const uint32_t yb = it & 1u;
        if (!mbar_wait(smem_u32(&yfull[yb]), (it >> 1) & 1u, abort, a.status)) break;
        tc_fence_after();
        const uint32_t ybase = smem_u32(ybuf_s + yb * YB);
        for (int j = 0; j < w.nchunks; ++j, ++cc) {
          const uint32_t slot = cc % kWbSlots;
          if (!mbar_wait(smem_u32(&dempty[slot]), ((cc / kWbSlots) & 1u) ^ 1u, abort, a.status)) { ok = false; break; }
          const uint32_t st = consumed % S, ph = (consumed / S) & 1u;
          if (!mbar_wait(smem_u32(&full[st]), ph, abort, a.status)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sx = smem_u32(ring + st * kStage);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint64_t ad = cols ? desc_kmajor_sw128(sx + (kk >> 2) * kBox + (kk & 3) * 32u)
                                         : desc_mnmajor_sw128_2atoms(sx + kk * 2048u, kBox);
            const uint64_t bd = desc_kmajor_sw128(ybase + (kk >> 2) * (YB / 2) + (kk & 3) * 32u);
            umma_bf16(tmem + slot * NZ, ad, bd, idesc, kk > 0 ? 1u : 0u);
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
    const int nheads = GPT * G;  // head slots per key tile (<= NZ / 2)
    const int units = nheads * (DH / 8);
    uint32_t staged = 0;
    // Stage Y (hi/lo bf16, swizzled K-major) of item t into buffer staged & 1.
    auto stage = [&](int t) -> bool {
      const WbItem w = decode_item(s, t);
      const uint32_t yb = staged & 1u;
      const bool ok = mbar_wait(smem_u32(&yempty[yb]), ((staged >> 1) & 1u) ^ 1u, abort, a.status);
      if (ok) {
        uint8_t* ybase = ybuf_s + yb * YB;
        for (int unit = ethr; unit < units; unit += 128) {
          const int u = unit / (DH / 8);                  // head slot gi*G + j
          const int i0 = (unit - u * (DH / 8)) * 8;
          const int gi = u / G;
          const int g = w.tile * GPT + gi;
          float v[8];
          if (g < s.nkv) {
            const float* src = a.ybuf + (static_cast<size_t>(w.layer) * s.nq + g * G + (u - gi * G)) * DH + i0;
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
            split_hilo(v[e], f16, hb[e], lb[e]);
          }
          const int k = gi * DH + i0;                     // K index of the 8-element chunk
          const int region = k >> 6, chunk = (k & 63) >> 3;
          const int rhi = u, rlo = NZ / 2 + u;
          uint8_t* base = ybase + region * (YB / 2);
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
    // y (and the caller's v_in, which v_out may alias) belong to the kernel launched
    // before this one: wait until it has completed.  The producer's W^K copies and the
    // prologue do not depend on it and may already run.
    griddep_wait();
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
        const uint32_t taddr = tmem + (static_cast<uint32_t>(q * 32) << 16) + slot * NZ;
        const int col = w.c0 + 128 * j + q * 32 + lane;
#pragma unroll
        for (int n0 = 0; n0 < NZ / 2; n0 += 16) {  // hi rows n0.., lo rows NZ/2 + n0..
          uint32_t hi[16], lo[16];
          tmem_ld16(taddr + n0, hi);
          tmem_ld16(taddr + NZ / 2 + n0, lo);
          tmem_ld_wait();
          if (col < s.d) {
#pragma unroll
            for (int e = 0; e < 16; ++e) {
              const int u = n0 + e;
              if (u < nheads) {
                const int gi = u / G;
                const int g = w.tile * GPT + gi;
                if (g < s.nkv) {
                  const size_t h = static_cast<size_t>(w.layer) * s.nq + g * G + (u - gi * G);
                  a.v_out[h * s.d + col] = __uint_as_float(hi[e]) + __uint_as_float(lo[e]);
                }
              }
            }
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
    tmem_dealloc(tmem, Cfg::kTmemCols);
  }
}

template <int DH, int NZ, bool GENERIC>
cudaError_t launch_wb_gen(const WbArgs& a, int num_sms, cudaStream_t st) {
  using Cfg = WbCfg<NZ>;
  static unsigned long long configured = 0;  // one bit per device: the attribute is per device
  cudaError_t e = set_smem_per_device(reinterpret_cast<const void*>(writeback_kernel<DH, NZ, GENERIC>),
                                      static_cast<int>(Cfg::kSmem), configured);
  if (e != cudaSuccess) return e;
  const int ncb = (a.s.d + kWbCols - 1) / kWbCols;
  const int T = a.s.L * a.s.tiles_k * ncb;
  const int grid = T < num_sms ? T : num_sms;
  // Programmatic dependent launch: the CTAs may start as the previous kernel's CTAs exit
  // (only the reads of y wait for that kernel, see griddep_wait).
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kWbThreads);
  cfg.dynamicSmemBytes = Cfg::kSmem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, writeback_kernel<DH, NZ, GENERIC>, a);
  if (e == cudaErrorNotSupported || e == cudaErrorInvalidValue) {
    (void)cudaGetLastError();  // the attribute is refused here: an ordinary stream-ordered launch
    writeback_kernel<DH, NZ, GENERIC><<<grid, kWbThreads, Cfg::kSmem, st>>>(a);
  }
  return cudaGetLastError();
}

template <int DH, int NZ>
cudaError_t launch_wb_cfg(const WbArgs& a, int num_sms, cudaStream_t st) {
  return (a.s.cols || a.s.f16) ? launch_wb_gen<DH, NZ, true>(a, num_sms, st) : launch_wb_gen<DH, NZ, false>(a, num_sms, st);
}

template <int DH>
cudaError_t launch_wb_dh(const WbArgs& a, int num_sms, cudaStream_t st) {
  switch (a.s.nz) {
    case 16: return launch_wb_cfg<DH, 16>(a, num_sms, st);
    case 32: return launch_wb_cfg<DH, 32>(a, num_sms, st);
    case 64: return launch_wb_cfg<DH, 64>(a, num_sms, st);
    case 128: return launch_wb_cfg<DH, 128>(a, num_sms, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_writeback(const WbArgs& a, int num_sms, cudaStream_t st) {
  if (a.s.dh == 128) return launch_wb_dh<128>(a, num_sms, st);
  if (a.s.dh == 64) return launch_wb_dh<64>(a, num_sms, st);
  return cudaErrorInvalidValue;
}

}  // namespace gas
