// Whole-layer spectral norm (Section 4.2, Appendix E): sigma_l = ||M||_2 for the layer's
// full interaction matrix M = W^Q W^K_exp^T, every query head at once, by power iteration
// on M with one persistent v per layer.  W^K_exp = W^K R^T, where R (n_q d_h x n_kv d_h)
// repeats each KV group's d_h coordinates for its G query heads, so W^K is never expanded:
//
//   M v   = W^Q (R (W^K^T v)):   a row-dot pass over Wk (n_kv*d_h values), the G-fold
//                                repeat, then a column-sum pass over Wq (d values)
//   M^T u = W^K (R^T (W^Q^T u)): a row-dot pass over Wq (n_q*d_h values), R^T sums the G
//                                query blocks of each group, then a column-sum pass over Wk
//
// with sigma = ||M v|| and v <- M^T u / ||M^T u|| for u = M v / ||M v||.
//
// In the nn.Linear layout Wq[r][c] (r < n_q*d_h, c < d) is W^Q[c][r], so W^Q^T x is a row
// dot product and W^Q z a column sum.  The z-space has n_q*d_h dimensions, too many for
// the d_h x d_h Gram reduction of the per-head path, so every iteration streams each
// matrix twice.  Normalisations are recomputed by the consumer of a vector from the
// full vector (d floats), so no partial norms have to travel between kernels.

#include "gas_device.cuh"

namespace gas {

namespace {

constexpr int kRowBlock = 64;  // rows per rowdot CTA (8 warps x 8 rows)

// 8 weights of row r at column c (zero beyond the matrix) and their dot with x[c .. c+8).
template <int WT>
__device__ __forceinline__ float dot8(const W8<WT>& q, const float* xs, int c) {
  const float4 x0 = *reinterpret_cast<const float4*>(xs + c);
  const float4 x1 = *reinterpret_cast<const float4*>(xs + c + 4);
  float f[8];
  unpack_w8<WT>(q, f);
  float t = f[0] * x0.x;
  t = fmaf(f[1], x0.y, t); t = fmaf(f[2], x0.z, t); t = fmaf(f[3], x0.w, t);
  t = fmaf(f[4], x1.x, t); t = fmaf(f[5], x1.y, t); t = fmaf(f[6], x1.z, t);
  return fmaf(f[7], x1.w, t);
}

// out[l][r] = sum_c W_l[r][c] * x_l[c] / ||x_l|| for a block of 64 rows (d values of x).
// x is staged unnormalised while its squared norm is summed, and the 64 results are
// scaled at the end.  Each lane keeps 16 weight loads in flight (8 rows x 2 column
// blocks of 256).
template <int WT>
__global__ void __launch_bounds__(256) layer_rowdot_kernel(const __grid_constant__ LayerTable tab,
                                                           const __grid_constant__ LayerArgs a) {
  extern __shared__ float lsm[];
  float* xs = lsm;            // [d]
  float* red = lsm + a.s.d;   // [8]
  const int l = blockIdx.y;
  const bool isq = a.which == 1;
  const int R = (isq ? a.s.nq : a.s.nkv) * a.s.dh;
  const int d = a.s.d;
  const void* W = isq ? tab.q[l] : tab.k[l];
  const long long ld = isq ? a.s.ldq : a.s.ldk;
  const long long hstride = isq ? a.s.hsq : a.s.hsk;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  {
    const float* src = a.src + static_cast<size_t>(l) * d;
    float n2 = 0.0f;
    for (int i = threadIdx.x * 4; i < d; i += blockDim.x * 4) {
      const float4 v = *reinterpret_cast<const float4*>(src + i);
      n2 = fmaf(v.x, v.x, fmaf(v.y, v.y, fmaf(v.z, v.z, fmaf(v.w, v.w, n2))));
      *reinterpret_cast<float4*>(xs + i) = v;
    }
    n2 = warp_sum(n2);
    if (lane == 0) red[warp] = n2;
    __syncthreads();
  }
  float n2 = 0.0f;
#pragma unroll
  for (int w = 0; w < 8; ++w) n2 += red[w];
  const float inv = safe_inv_sqrt(n2);
  const int r0 = blockIdx.x * kRowBlock + warp * 8;
  long long roff[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) roff[i] = weight_row_offset(r0 + i < R ? r0 + i : r0, a.s.dh, ld, hstride);
  float acc[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) acc[i] = 0.0f;
  for (int c = lane * 8; c < d; c += 512) {
    const int c2 = c + 256;
    const bool two = c2 < d;
    W8<WT> q0[8], q1[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const bool ok = r0 + i < R;
      q0[i] = ok ? load_w8<WT>(W, roff[i] + c) : zero_w8<WT>();
      q1[i] = (ok && two) ? load_w8<WT>(W, roff[i] + c2) : zero_w8<WT>();
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      acc[i] += dot8<WT>(q0[i], xs, c);
      if (two) acc[i] += dot8<WT>(q1[i], xs, c2);
    }
  }
  int idx;
  const float tot = warp_transpose_reduce<8>(acc, lane, idx);
  if (transpose_reduce_writer<8>(lane) && r0 + idx < R)
    a.out[static_cast<size_t>(l) * a.out_stride + r0 + idx] = tot * inv;
}

// out[l][c] = sum_r W_l[r][c] * x_l[r] for a chunk of 256 columns over all rows, with
// x = RepeatBlocks(src) (query matrix) or SumGroups(src) (key matrix).
template <int WT>
__global__ void __launch_bounds__(256) layer_coldot_kernel(const __grid_constant__ LayerTable tab,
                                                           const __grid_constant__ LayerArgs a) {
  extern __shared__ float lsm[];
  const Shape& s = a.s;
  const int l = blockIdx.y;
  const bool isq = a.which == 1;
  const int R = (isq ? s.nq : s.nkv) * s.dh;
  const void* W = isq ? tab.q[l] : tab.k[l];
  const long long ld = isq ? s.ldq : s.ldk;
  const long long hstride = isq ? s.hsq : s.hsk;
  float* xs = lsm;                  // [R]
  float* red = lsm + R;             // [8][256]
  const float* src = a.src + static_cast<size_t>(l) * a.src_stride;
  for (int r = threadIdx.x; r < R; r += blockDim.x) {
    const int i = r % s.dh;
    if (isq) {  // RepeatBlocks(z_kv, G): query row block h reads key block h / G
      const int hq = r / s.dh;
      xs[r] = src[(hq / s.G) * s.dh + i];
    } else {    // SumGroups(y, G): key row block g sums query blocks g*G .. g*G+G-1
      const int g = r / s.dh;
      float acc = 0.0f;
      for (int j = 0; j < s.G; ++j) acc += src[(g * s.G + j) * s.dh + i];
      xs[r] = acc;
    }
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c = blockIdx.x * 256 + lane * 8;
  float acc[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) acc[e] = 0.0f;
  if (c < s.d) {
    // warp w takes rows w, w + 8, ...; eight of them are loaded before any is used
    int r = warp;
    for (; r + 56 < R; r += 64) {
      W8<WT> q[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) q[j] = load_w8<WT>(W, weight_row_offset(r + 8 * j, s.dh, ld, hstride) + c);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        float f[8];
        unpack_w8<WT>(q[j], f);
        const float xr = xs[r + 8 * j];
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] = fmaf(f[e], xr, acc[e]);
      }
    }
    for (; r < R; r += 8) {
      const W8<WT> q = load_w8<WT>(W, weight_row_offset(r, s.dh, ld, hstride) + c);
      float f[8];
      unpack_w8<WT>(q, f);
      const float xr = xs[r];
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] = fmaf(f[e], xr, acc[e]);
    }
  }
  float4* rp = reinterpret_cast<float4*>(&red[warp * 256 + lane * 8]);
  rp[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
  rp[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
  __syncthreads();
  const int cc = blockIdx.x * 256 + threadIdx.x;
  if (cc < s.d) {
    float tot = 0.0f;
#pragma unroll
    for (int w = 0; w < 8; ++w) tot += red[w * 256 + threadIdx.x];
    a.out[static_cast<size_t>(l) * a.out_stride + cc] = tot;
  }
}

// sigma_l = ||u'_l|| of the last iteration; v_out = v'/||v'||; fused scale (Eq. 15).
__global__ void __launch_bounds__(256) layer_finalize_kernel(const __grid_constant__ LayerArgs a) {
  __shared__ float red[8];
  const Shape& s = a.s;
  const int l = blockIdx.x;
  const float* u = a.src + static_cast<size_t>(l) * s.d;
  float n2 = 0.0f;
  for (int i = threadIdx.x * 4; i < s.d; i += blockDim.x * 4) {
    const float4 v = *reinterpret_cast<const float4*>(u + i);
    n2 = fmaf(v.x, v.x, fmaf(v.y, v.y, fmaf(v.z, v.z, fmaf(v.w, v.w, n2))));
  }
  n2 = warp_sum(n2);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = n2;
  __syncthreads();
  float tot = 0.0f;
  for (int w = 0; w < 8; ++w) tot += red[w];
  const float sigma = sqrtf(tot);
  if (a.v_out != nullptr) {
    __syncthreads();
    const float* vp = a.vsrc + static_cast<size_t>(l) * s.d;
    float m2 = 0.0f;
    for (int i = threadIdx.x * 4; i < s.d; i += blockDim.x * 4) {
      const float4 v = *reinterpret_cast<const float4*>(vp + i);
      m2 = fmaf(v.x, v.x, fmaf(v.y, v.y, fmaf(v.z, v.z, fmaf(v.w, v.w, m2))));
    }
    m2 = warp_sum(m2);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m2;
    __syncthreads();
    float mt = 0.0f;
    for (int w = 0; w < 8; ++w) mt += red[w];
    const float inv = safe_inv_sqrt(mt);
    float* vo = a.v_out + static_cast<size_t>(l) * s.d;
    for (int i = threadIdx.x * 4; i < s.d; i += blockDim.x * 4) {
      float4 v = *reinterpret_cast<const float4*>(vp + i);
      v.x *= inv; v.y *= inv; v.z *= inv; v.w *= inv;
      *reinterpret_cast<float4*>(vo + i) = v;
    }
  }
  if (threadIdx.x == 0) {
    a.sigma[l] = sigma;
    if (!isfinite(sigma)) set_status(a.status, GAS_DEV_NONFINITE_SIGMA);
    if (a.scale_out != nullptr) a.scale_out[l] = a.scale_c * sigma;
  }
}

}  // namespace

template <int WT>
cudaError_t launch_rowdot_dt(const LayerTable& tab, const LayerArgs& a, cudaStream_t st) {
  const int R = (a.which == 1 ? a.s.nq : a.s.nkv) * a.s.dh;
  const dim3 grid((R + kRowBlock - 1) / kRowBlock, a.s.L);
  const size_t smem = (a.s.d + 8) * sizeof(float);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(layer_rowdot_kernel<WT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  layer_rowdot_kernel<WT><<<grid, 256, smem, st>>>(tab, a);
  return cudaGetLastError();
}

template <int WT>
cudaError_t launch_coldot_dt(const LayerTable& tab, const LayerArgs& a, cudaStream_t st) {
  const int R = (a.which == 1 ? a.s.nq : a.s.nkv) * a.s.dh;
  const dim3 grid((a.s.d + 255) / 256, a.s.L);
  const size_t smem = (R + 8 * 256) * sizeof(float);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(layer_coldot_kernel<WT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  layer_coldot_kernel<WT><<<grid, 256, smem, st>>>(tab, a);
  return cudaGetLastError();
}

cudaError_t launch_layer_rowdot(const LayerTable& tab, const LayerArgs& a, cudaStream_t st) {
  return a.s.f32 ? launch_rowdot_dt<kWF32>(tab, a, st)
                 : a.s.f16 ? launch_rowdot_dt<kWF16>(tab, a, st) : launch_rowdot_dt<kWBf16>(tab, a, st);
}

cudaError_t launch_layer_coldot(const LayerTable& tab, const LayerArgs& a, cudaStream_t st) {
  return a.s.f32 ? launch_coldot_dt<kWF32>(tab, a, st)
                 : a.s.f16 ? launch_coldot_dt<kWF16>(tab, a, st) : launch_coldot_dt<kWBf16>(tab, a, st);
}

cudaError_t launch_layer_finalize(const LayerArgs& a, cudaStream_t st) {
  layer_finalize_kernel<<<a.s.L, 256, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace gas
