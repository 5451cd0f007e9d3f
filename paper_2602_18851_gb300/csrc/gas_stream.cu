// Streaming matvec-chain back end: Algorithm 2 (Appendix E.1) applied literally,
// with the GQA key block read once per group (Algorithm 3, Section 4.2).
//
// One power iteration for head h (group g) is two weight passes:
//   Q pass over A_h = (W^Q_h)^T:  u' = A_h^T z (per column chunk), ||u'||^2, t = A_h u'
//   K pass over B_g = (W^K_g)^T:  y = t/||u'||;  v' = B_g^T y, ||v'||^2, z_next = B_g v'
// (z = B_g v for the normalised v, so z_next must be divided by ||v'||; the next Q
// pass does that when it reads it).  The start is a K0 pass z = B_g v_in with
// ||v_in||^2, and the last K pass writes v' itself (normalised by the finalize kernel).
// Each CTA streams one d_h x 256 weight tile (bf16, binary16 or fp32; any d_h in
// {64, 80, 96, 128, 256}) with 16-byte loads, issued before anything else, and stages
// its input vectors (one, or the G of a key group) in shared memory while they land.
// Its results over its columns go to a small fp32 workspace indexed by chunk; a second,
// short kernel sums them in chunk order into one d_h-vector and one squared norm per
// head.  No float atomics: results are deterministic.  In a Q pass every CTA also
// prefetches into L2 the tile of the CTA one wave after it, which then loads from L2.

#include "gas_device.cuh"

namespace gas {

namespace {

// Smallest power of two >= x (the warp transpose-reduction works on 2^n values).
__host__ __device__ constexpr int pow2_at_least(int x) { return x <= 1 ? 1 : 2 * pow2_at_least((x + 1) / 2); }

// Warps per CTA: 8, or 16 for d_h 256 so that every thread holds at most 16 rows.
__host__ __device__ constexpr int stream_warps(int dh) { return dh > 128 ? 16 : 8; }

constexpr int kStreamVB = 8;  // input vectors staged in shared memory at a time

// Two CTAs per SM for 16-bit weights (one tile loading while the other reduces); fp32
// tiles need twice the registers.
template <int DH, int MODE, int WT>
__global__ void __launch_bounds__(32 * stream_warps(DH), (WT == kWF32 || DH > 128) ? 1 : 2)
    stream_pass_kernel(const __grid_constant__ LayerTable tab,
                                                                            const __grid_constant__ StreamArgs a) {
  constexpr int NW = stream_warps(DH);
  constexpr int NT = 32 * NW;
  constexpr int RV = DH / NW;             // rows held per thread (warp w owns rows w, w+NW, ...)
  constexpr int R = pow2_at_least(RV);    // padded to a power of two with zero rows
  const Shape& s = a.s;
  const int chunk = blockIdx.x, m = blockIdx.y, l = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int col = chunk * kStreamChunk + lane * 8;
  const bool colok = col < s.d;  // d % 8 == 0: a lane's 8 columns are all in or all out
  const long long ld = (MODE == kPassQ) ? s.ldq : s.ldk;
  const long long hstride = (MODE == kPassQ) ? s.hsq : s.hsk;
  const void* X = (MODE == kPassQ) ? tab.q[l] : tab.k[l];
  const long long x0 = static_cast<long long>(m) * hstride;

  W8<WT> w[R];
#pragma unroll
  for (int rr = 0; rr < R; ++rr) {
    const int row = warp + NW * rr;
    w[rr] = (rr < RV && colok) ? load_w8<WT>(X, x0 + static_cast<long long>(row) * ld + col) : zero_w8<WT>();
  }
  // Bring into L2 the tile of the CTA a.pf_dist positions later in launch order (about one
  // wave ahead): when that CTA runs, its loads hit L2, so a CTA spends less of its life
  // waiting and more of the SM's time has weights in flight.
  if (a.pf_dist > 0) {
    const long long lin = blockIdx.x + static_cast<long long>(gridDim.x) * (blockIdx.y + static_cast<long long>(gridDim.y) * blockIdx.z);
    const long long fut = lin + a.pf_dist;
    const long long total = static_cast<long long>(gridDim.x) * gridDim.y * gridDim.z;
    if (fut < total) {
      const int fc = static_cast<int>(fut % gridDim.x);
      const long long fr = fut / gridDim.x;
      const int fm = static_cast<int>(fr % gridDim.y), fl = static_cast<int>(fr / gridDim.y);
      const int fcol = fc * kStreamChunk + lane * 8;
      if (fcol < s.d) {
        const char* FX = reinterpret_cast<const char*>((MODE == kPassQ) ? tab.q[fl] : tab.k[fl]);
        const long long fx0 = static_cast<long long>(fm) * hstride;
#pragma unroll
        for (int rr = 0; rr < RV; ++rr) {
          const long long e = fx0 + static_cast<long long>(warp + NW * rr) * ld + fcol;
          asm volatile("prefetch.global.L2 [%0];" ::"l"(FX + e * (WT == kWF32 ? 4 : 2)));
        }
      }
    }
  }

  __shared__ __align__(16) float xs[kStreamVB][DH];
  __shared__ __align__(16) float red[NW][kStreamChunk];
  __shared__ __align__(16) float ps[kStreamChunk];

  const int nvec = (MODE == kPassQ) ? 1 : s.G;
  const size_t h0 = static_cast<size_t>(l) * s.nq + ((MODE == kPassQ) ? m : m * s.G);  // head of vector 0
  for (int j0 = 0; j0 < nvec; j0 += kStreamVB) {
    const int nb = min(kStreamVB, nvec - j0);
    if (MODE != kPassK0) {
      if (j0 > 0) __syncthreads();  // every thread is done with the previous batch
      for (int i = tid; i < nb * DH; i += NT) {
        const int jj = i / DH, r = i - jj * DH;
        const size_t hidx = h0 + j0 + jj;
        float x = __ldg(a.in + hidx * DH + r);
        if (a.in_scaled) x *= safe_inv_sqrt(__ldg(a.in2 + hidx));
        xs[jj][r] = x;
      }
      __syncthreads();
    }
    for (int jj = 0; jj < nb; ++jj) {
      const size_t hidx = h0 + j0 + jj;
      float p[8];
      if (MODE == kPassK0) {
        if (colok) {
          const float4* vp = reinterpret_cast<const float4*>(a.v_in + hidx * s.d + col);
          const float4 v0 = __ldg(vp), v1 = __ldg(vp + 1);
          p[0] = v0.x; p[1] = v0.y; p[2] = v0.z; p[3] = v0.w;
          p[4] = v1.x; p[5] = v1.y; p[6] = v1.z; p[7] = v1.w;
        } else {
#pragma unroll
          for (int c = 0; c < 8; ++c) p[c] = 0.0f;
        }
      } else {
        // p = X^T x over this chunk: per-warp partials over its rows, then summed
        float pp[8];
#pragma unroll
        for (int c = 0; c < 8; ++c) pp[c] = 0.0f;
#pragma unroll
        for (int rr = 0; rr < RV; ++rr) {
          float f[8];
          unpack_w8<WT>(w[rr], f);
          const float xr = xs[jj][warp + NW * rr];
#pragma unroll
          for (int c = 0; c < 8; ++c) pp[c] = fmaf(f[c], xr, pp[c]);
        }
        float4* rp = reinterpret_cast<float4*>(&red[warp][lane * 8]);
        rp[0] = make_float4(pp[0], pp[1], pp[2], pp[3]);
        rp[1] = make_float4(pp[4], pp[5], pp[6], pp[7]);
        __syncthreads();
        if (tid < kStreamChunk) {
          float tot = 0.0f;
          for (int ww = 0; ww < NW; ++ww) tot += red[ww][tid];
          ps[tid] = tot;
        }
        __syncthreads();
        const float4* pq = reinterpret_cast<const float4*>(&ps[lane * 8]);
        const float4 p0 = pq[0], p1 = pq[1];
        p[0] = p0.x; p[1] = p0.y; p[2] = p0.z; p[3] = p0.w;
        p[4] = p1.x; p[5] = p1.y; p[6] = p1.z; p[7] = p1.w;
      }

      if (warp == 0) {  // each warp's lanes span the whole chunk: warp 0 owns ||p||^2
        float q2 = 0.0f;
#pragma unroll
        for (int c = 0; c < 8; ++c) q2 = fmaf(p[c], p[c], q2);
        q2 = warp_sum(q2);
        if (lane == 0) a.out2[hidx * s.nch + chunk] = q2;
        if (MODE == kPassKOut && colok) {
          float4* vo = reinterpret_cast<float4*>(a.v_out + hidx * s.d + col);
          vo[0] = make_float4(p[0], p[1], p[2], p[3]);
          vo[1] = make_float4(p[4], p[5], p[6], p[7]);
        }
      }
      if (MODE != kPassKOut) {
        float qv[R];
#pragma unroll
        for (int rr = 0; rr < R; ++rr) {
          float f[8];
          unpack_w8<WT>(w[rr], f);
          float acc = 0.0f;
#pragma unroll
          for (int c = 0; c < 8; ++c) acc = fmaf(f[c], p[c], acc);
          qv[rr] = acc;
        }
        int idx;
        const float r = warp_transpose_reduce<R>(qv, lane, idx);
        if (transpose_reduce_writer<R>(lane) && idx < RV)
          a.out[(hidx * s.nch + chunk) * DH + warp + NW * idx] = r;
      }
    }
  }
  if (MODE == kPassK0 && a.s_zero != nullptr && chunk == 0 && m == 0 && tid == 0) a.s_zero[l] = 0.0f;
}

// Sums of the chunk partials of a pass, in chunk order: outr[h] = sum_c out[h][c] (modes Q,
// K, K0) and outr2[h] = sum_c out2[h][c] (all modes), one thread per output value.  A
// separate launch: the pass's CTAs write their partials and exit without a fence or a
// ticket, so none of them waits for its stores to be acknowledged.
template <int DH>
__global__ void __launch_bounds__(256) stream_reduce_kernel(const __grid_constant__ StreamArgs a) {
  const Shape& s = a.s;
  const size_t heads = static_cast<size_t>(s.L) * s.nq;
  const int nch = s.nch;
  const size_t i = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (a.mode != kPassKOut && i < heads * DH) {
    const size_t hidx = i / DH, r = i - hidx * DH;
    const float* src = a.out + hidx * nch * DH + r;
    float acc[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = 0.0f;
    for (int c0 = 0; c0 < nch; c0 += 8) {  // eight loads in flight per step
      float t[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) t[e] = c0 + e < nch ? __ldcg(src + static_cast<size_t>(c0 + e) * DH) : 0.0f;
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] += t[e];
    }
    a.outr[i] = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
  }
  if (i < heads) {
    const float* src = a.out2 + i * nch;
    float v = 0.0f;
    for (int c = 0; c < nch; ++c) v += __ldcg(src + c);
    a.outr2[i] = v;
  }
}

// sigma = ||u'|| of the last Q pass; v_out = v' / ||v'|| of the last K pass; fused
// per-layer max of the scale (Eq. 15) by an atomic max on non-negative float bits.
__global__ void __launch_bounds__(256) finalize_kernel(const __grid_constant__ FinalizeArgs a) {
  const Shape& s = a.s;
  const size_t hidx = blockIdx.x;
  const int l = static_cast<int>(hidx / s.nq);
  const float sigma = sqrtf(a.s2[hidx]);
  if (a.v_out != nullptr) {
    const float inv = safe_inv_sqrt(a.n2[hidx]);
    float4* v = reinterpret_cast<float4*>(a.v_out + hidx * s.d);
    for (int i = threadIdx.x; i < s.d / 4; i += blockDim.x) {
      float4 x = v[i];
      x.x *= inv; x.y *= inv; x.z *= inv; x.w *= inv;
      v[i] = x;
    }
  }
  if (threadIdx.x == 0) {
    a.sigma[hidx] = sigma;
    if (!isfinite(sigma)) set_status(a.status, GAS_DEV_NONFINITE_SIGMA);
    if (a.scale_out != nullptr) atomic_max_nonneg(&a.scale_out[l], a.scale_c * sigma);
  }
}

__device__ __forceinline__ float nanmax(float a, float b) { return (b != b || b > a) ? b : a; }

// Eq. 15 per layer: s[l] = c * max_h sigma[l][h] (a NaN sigma propagates).
__global__ void __launch_bounds__(32) scales_kernel(const __grid_constant__ ScalesArgs a) {
  const int l = blockIdx.x;
  float m = 0.0f;
  for (int h = threadIdx.x; h < a.nq; h += 32) m = nanmax(m, a.sigma[static_cast<size_t>(l) * a.nq + h]);
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) m = nanmax(m, __shfl_xor_sync(0xFFFFFFFFu, m, off));
  if (threadIdx.x == 0) a.s[l] = a.scale_c * m;
}

// Streaming multiprocessors of the current device (looked up once per device).
int current_sm_count() {
  static int counts[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 0;
  if (dev < 64 && __atomic_load_n(&counts[dev], __ATOMIC_RELAXED) > 0) return __atomic_load_n(&counts[dev], __ATOMIC_RELAXED);
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  if (dev < 64) __atomic_store_n(&counts[dev], n, __ATOMIC_RELAXED);
  return n;
}

template <int DH, int WT>
cudaError_t launch_stream_dt(const LayerTable& tab, const StreamArgs& a_in, cudaStream_t st) {
  // Q passes (one vector per tile, bound by the weight stream) prefetch the tile of the CTA
  // one wave later into L2; key passes (G vectors per tile, bound by the SM) do not.
  StreamArgs a = a_in;
  a.pf_dist = a.mode == kPassQ ? static_cast<long long>(current_sm_count()) * ((WT == kWF32 || DH > 128) ? 1 : 2) : 0;
  const dim3 block(32 * stream_warps(DH));
  const dim3 grid(a.s.nch, a.mode == kPassQ ? a.s.nq : a.s.nkv, a.s.L);
  switch (a.mode) {
    case kPassQ: stream_pass_kernel<DH, kPassQ, WT><<<grid, block, 0, st>>>(tab, a); break;
    case kPassK: stream_pass_kernel<DH, kPassK, WT><<<grid, block, 0, st>>>(tab, a); break;
    case kPassK0: stream_pass_kernel<DH, kPassK0, WT><<<grid, block, 0, st>>>(tab, a); break;
    case kPassKOut: stream_pass_kernel<DH, kPassKOut, WT><<<grid, block, 0, st>>>(tab, a); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

template <int DH>
cudaError_t launch_stream_dh(const LayerTable& tab, const StreamArgs& a, cudaStream_t st) {
  if (a.s.f32) {
    if (DH > 128) return cudaErrorInvalidValue;  // fp32 rows of d_h 256 do not fit the registers
    return launch_stream_dt<(DH > 128 ? 128 : DH), kWF32>(tab, a, st);
  }
  return a.s.f16 ? launch_stream_dt<DH, kWF16>(tab, a, st) : launch_stream_dt<DH, kWBf16>(tab, a, st);
}

}  // namespace

cudaError_t launch_stream_pass(const LayerTable& tab, const StreamArgs& a, cudaStream_t st) {
  switch (a.s.dh) {
    case 64: return launch_stream_dh<64>(tab, a, st);
    case 80: return launch_stream_dh<80>(tab, a, st);
    case 96: return launch_stream_dh<96>(tab, a, st);
    case 128: return launch_stream_dh<128>(tab, a, st);
    case 256: return launch_stream_dh<256>(tab, a, st);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_stream_reduce(const StreamArgs& a, cudaStream_t st) {
  const int dh = a.s.dh;
  const size_t outs = static_cast<size_t>(a.s.L) * a.s.nq * (a.mode == kPassKOut ? 1 : dh);
  const unsigned grid = static_cast<unsigned>((outs + 255) / 256);
  switch (dh) {
    case 64: stream_reduce_kernel<64><<<grid, 256, 0, st>>>(a); break;
    case 80: stream_reduce_kernel<80><<<grid, 256, 0, st>>>(a); break;
    case 96: stream_reduce_kernel<96><<<grid, 256, 0, st>>>(a); break;
    case 128: stream_reduce_kernel<128><<<grid, 256, 0, st>>>(a); break;
    case 256: stream_reduce_kernel<256><<<grid, 256, 0, st>>>(a); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t launch_finalize(const FinalizeArgs& a, cudaStream_t st) {
  finalize_kernel<<<a.s.L * a.s.nq, 256, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_scales(const ScalesArgs& a, cudaStream_t st) {
  scales_kernel<<<a.L, 32, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace gas
