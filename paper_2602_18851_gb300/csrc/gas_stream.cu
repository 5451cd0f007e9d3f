// Streaming matvec-chain back end: Algorithm 2 (Appendix E.1) applied literally,
// with the GQA key block read once per group (Algorithm 3, Section 4.2).
//
// One power iteration for head h (group g) is two weight passes:
//   Q pass over A_h = (W^Q_h)^T:  u' = A_h^T z (per column chunk), ||u'||^2, t = A_h u'
//   K pass over B_g = (W^K_g)^T:  y = t/||u'||;  v' = B_g^T y, ||v'||^2, z_next = B_g v'
// (z = B_g v for the normalised v, so z_next must be divided by ||v'||; the consumer
// does that when it sums the partials).  The start is a K0 pass z = B_g v_in with
// ||v_in||^2, and the last K pass writes v' itself (normalised by the finalize kernel).
// Each CTA streams one d_h x 256 weight tile (bf16, binary16 or fp32; any d_h in
// {64, 80, 96, 128, 256}) with 16-byte loads; partial results over
// its columns go to a small fp32 workspace indexed by chunk and are summed, in a fixed
// order, by the next pass (no atomics, deterministic).

#include "gas_device.cuh"

namespace gas {

namespace {

// Smallest power of two >= x (the warp transpose-reduction works on 2^n values).
__host__ __device__ constexpr int pow2_at_least(int x) { return x <= 1 ? 1 : 2 * pow2_at_least((x + 1) / 2); }

// Warps per CTA: 8, or 16 for d_h 256 so that every thread holds at most 16 rows.
__host__ __device__ constexpr int stream_warps(int dh) { return dh > 128 ? 16 : 8; }

template <int DH, int MODE, int WT>
__global__ void __launch_bounds__(32 * stream_warps(DH)) stream_pass_kernel(const __grid_constant__ LayerTable tab,
                                                                            const __grid_constant__ StreamArgs a) {
  constexpr int NW = stream_warps(DH);
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

  __shared__ float xs[DH];
  __shared__ __align__(16) float red[NW][kStreamChunk];
  __shared__ __align__(16) float ps[kStreamChunk];

  const int nvec = (MODE == kPassQ) ? 1 : s.G;
  for (int j = 0; j < nvec; ++j) {
    const int h = (MODE == kPassQ) ? m : m * s.G + j;
    const size_t hidx = static_cast<size_t>(l) * s.nq + h;
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
      __syncthreads();  // every thread is done with xs / ps of the previous vector
      if (tid < DH) {
        float acc = 0.0f;
        for (int ch = 0; ch < a.in_nch; ++ch) acc += a.in[(hidx * a.in_nch + ch) * DH + tid];
        if (a.in_scaled) {
          float n2 = 0.0f;
          for (int ch = 0; ch < a.in_nch; ++ch) n2 += a.in2[hidx * a.in_nch + ch];
          acc *= safe_inv_sqrt(n2);
        }
        xs[tid] = acc;
      }
      __syncthreads();
      float pp[8];
#pragma unroll
      for (int c = 0; c < 8; ++c) pp[c] = 0.0f;
#pragma unroll
      for (int rr = 0; rr < RV; ++rr) {
        float f[8];
        unpack_w8<WT>(w[rr], f);
        const float xr = xs[warp + NW * rr];
#pragma unroll
        for (int c = 0; c < 8; ++c) pp[c] = fmaf(f[c], xr, pp[c]);
      }
      float4* rp = reinterpret_cast<float4*>(&red[warp][lane * 8]);
      rp[0] = make_float4(pp[0], pp[1], pp[2], pp[3]);
      rp[1] = make_float4(pp[4], pp[5], pp[6], pp[7]);
      __syncthreads();
      float tot = 0.0f;
      if (tid < kStreamChunk) {
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
  if (MODE == kPassK0 && a.s_zero != nullptr && chunk == 0 && m == 0 && tid == 0) a.s_zero[l] = 0.0f;
}

// sigma = ||u'|| of the last Q pass; v_out = v' / ||v'|| of the last K pass; fused
// per-layer max of the scale (Eq. 15) by an atomic max on non-negative float bits.
__global__ void __launch_bounds__(256) finalize_kernel(const __grid_constant__ FinalizeArgs a) {
  const Shape& s = a.s;
  const size_t hidx = blockIdx.x;
  const int l = static_cast<int>(hidx / s.nq);
  float s2 = 0.0f, n2 = 0.0f;
  for (int ch = 0; ch < s.nch; ++ch) s2 += a.s2p[hidx * s.nch + ch];
  const float sigma = sqrtf(s2);
  if (a.v_out != nullptr) {
    for (int ch = 0; ch < s.nch; ++ch) n2 += a.n2p[hidx * s.nch + ch];
    const float inv = safe_inv_sqrt(n2);
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

template <int DH, int WT>
cudaError_t launch_stream_dt(const LayerTable& tab, const StreamArgs& a, cudaStream_t st) {
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

cudaError_t launch_finalize(const FinalizeArgs& a, cudaStream_t st) {
  finalize_kernel<<<a.s.L * a.s.nq, 256, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_scales(const ScalesArgs& a, cudaStream_t st) {
  scales_kernel<<<a.L, 32, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace gas
