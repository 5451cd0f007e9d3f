// The consumer side of a per-layer FP8 scale (include/gas_fp8.h).
//
//   fp8_quantize_kernel   Algorithm 1, Stage 3: S~ = S / scale -> E4M3 codes, with the
//                         per-call statistics of Table 4 (largest scaled logit, number of
//                         scaled logits beyond 448) and the step maximum max|S| that the
//                         delayed-scaling history (Eq. 1) and the slack ratio (Eq. 16) use.
//                         One streaming pass: 16 logits per thread and group (two or four
//                         16-byte loads, one 16-byte store of codes), four groups (bf16) or
//                         two (fp32) in flight per thread; per-CTA reductions
//                         go to a per-layer accumulator by atomics, and the last CTA to
//                         finish (ticket counter, no waiting) writes the statistics and
//                         clears the accumulator for the next call.
//   fp8_delayed_kernel    Eq. 1: max(history) / (448 eta) per layer.
//   fp8_end_step_kernel   history push; slack ratios of Eq. 16 during a burn-in.
//   fp8_auto_alpha_kernel Algorithm 4: sort the finite slack ratios on chip (bitonic
//                         network in shared memory), interpolate the q-quantile, times kappa.
//
// Division.  S / scale must be the IEEE float32 quotient, rounded to nearest, because the
// quotient decides the code.  With y = RN(1/scale) (one correctly rounded reciprocal per
// thread) each quotient is q0 = RN(S y), r = S - scale q0 (exact, one FMA) and
// q = RN(q0 + r y): Markstein's theorem (P. Markstein, IBM J. Res. Dev. 34(1), 1990)
// makes q the correctly rounded S / scale when no intermediate leaves the normal range.
// The library takes this path only when scale and 1/scale are normal; a quotient that
// overflows or is far beyond 448 keeps q0 (same sign, still an overflow), one in the
// subnormal range encodes to a signed zero either way (the sign is the IEEE sign of
// the quotient, taken from the operands).  Other scales use the compiler's division.

#include <cuda_fp8.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>

#include "../../include/gas_fp8.h"
#include "gas_device.cuh"

namespace {

constexpr int kThreads = 256;
constexpr float kRmax = 448.0f;

struct alignas(16) LayerAcc {
  unsigned amax_bits;       // max |S| bits (non-negative floats order like their bits; NaN on top)
  unsigned ticket;          // CTAs finished in the current call
  unsigned long long overflow;
};

struct QArgs {
  const void* s;
  long long n;
  const float* scale;
  uint8_t* q;
  LayerAcc* acc;
  unsigned* step_amax;
  gas_fp8_stats* stats;
};

// Two logits -> two codes (low byte = first).  Saturating: the cast saturates every
// finite or infinite overflow to +-448; NaN mode: overflowing quotients become NaN.
// The sign comes from the IEEE rule (XOR of the operand signs), so that a quotient
// that rounds to zero keeps it.
template <bool SAT>
__device__ __forceinline__ uint32_t encode2(float q0, float q1, unsigned& ovf) {
  const bool o0 = !(fabsf(q0) <= kRmax), o1 = !(fabsf(q1) <= kRmax);
  ovf += static_cast<unsigned>(o0) + static_cast<unsigned>(o1);
  if (!SAT) {
    q0 = o0 ? __int_as_float(0x7FC00000) : q0;
    q1 = o1 ? __int_as_float(0x7FC00000) : q1;
  }
  return static_cast<uint32_t>(__nv_cvt_float2_to_fp8x2(make_float2(q0, q1), __NV_SATFINITE, __NV_E4M3));
}

// Every NaN code as 0x7F (the cast may give either NaN pattern).
__device__ __forceinline__ uint32_t canon_nan4(uint32_t w) {
  uint32_t out = 0;
#pragma unroll
  for (int b = 0; b < 4; ++b) {
    uint32_t c = (w >> (8 * b)) & 0xFFu;
    if ((c & 0x7Fu) == 0x7Fu) c = 0x7Fu;
    out |= c << (8 * b);
  }
  return out;
}

// Sixteen logits as loaded: two 16-byte words of bf16, or four of fp32.
template <int DT>
struct Raw16 {
  uint4 w[DT == GAS_DTYPE_BF16 ? 2 : 4];
};

template <int DT>
__device__ __forceinline__ void load16(const QArgs& a, long long g, Raw16<DT>& r) {
  const uint4* p = reinterpret_cast<const uint4*>(a.s) + (DT == GAS_DTYPE_BF16 ? 2 : 4) * g;
#pragma unroll
  for (int i = 0; i < (DT == GAS_DTYPE_BF16 ? 2 : 4); ++i) r.w[i] = __ldcs(p + i);
}

// Widen sixteen loaded logits to fp32; returns their largest |x| as bits (non-negative
// floats order like their bit patterns; NaN above infinity).
template <int DT>
__device__ __forceinline__ uint32_t unpack16(const Raw16<DT>& r, float (&x)[16]) {
  if (DT == GAS_DTYPE_BF16) {
    const uint32_t w[8] = {r.w[0].x, r.w[0].y, r.w[0].z, r.w[0].w, r.w[1].x, r.w[1].y, r.w[1].z, r.w[1].w};
    __nv_bfloat162 m = __halves2bfloat162(__ushort_as_bfloat16(0), __ushort_as_bfloat16(0));
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t aw = w[i] & 0x7FFF7FFFu;
      m = __hmax2_nan(m, *reinterpret_cast<const __nv_bfloat162*>(&aw));
      x[2 * i] = gas::bf16lo(w[i]);
      x[2 * i + 1] = gas::bf16hi(w[i]);
    }
    const uint32_t mb = *reinterpret_cast<const uint32_t*>(&m);
    return max(mb << 16, mb & 0xFFFF0000u);
  } else {
    uint32_t m = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint32_t b[4] = {r.w[i].x, r.w[i].y, r.w[i].z, r.w[i].w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        x[4 * i + j] = __uint_as_float(b[j]);
        m = max(m, b[j] & 0x7FFFFFFFu);
      }
    }
    return m;
  }
}

// Codes of sixteen logits none of which overflows (every |x| below the threshold):
// the reciprocal-path quotient of |x| by a positive scale, then the sign of x.
__device__ __forceinline__ uint4 encode16_fast(const float (&x)[16], float sc, float y) {
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float q[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float ax = fabsf(x[4 * i + j]);
      const float q0 = ax * y;
      const float r = fmaf(-q0, sc, ax);
      const float qm = fmaf(r, y, q0);
      q[j] = __uint_as_float(__float_as_uint(qm) | (__float_as_uint(x[4 * i + j]) & 0x80000000u));
    }
    w[i] = static_cast<uint32_t>(__nv_cvt_float2_to_fp8x2(make_float2(q[0], q[1]), __NV_SATFINITE, __NV_E4M3)) |
           (static_cast<uint32_t>(__nv_cvt_float2_to_fp8x2(make_float2(q[2], q[3]), __NV_SATFINITE, __NV_E4M3))
            << 16);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// Codes of sixteen logits through the compiler's division, with overflow counting,
// NaN handling and the IEEE sign of every quotient (groups that reach the threshold,
// and every group when the scale is not a positive normal float).
template <bool SAT>
__device__ __forceinline__ uint4 encode16_exact(const float (&x)[16], float sc, unsigned& ovf) {
  const uint32_t sgn = __float_as_uint(sc) & 0x80000000u;
  uint32_t w[4];
  unsigned o = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float q[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float t = __fdiv_rn(x[4 * i + j], sc);
      q[j] = __uint_as_float((__float_as_uint(t) & 0x7FFFFFFFu) | ((__float_as_uint(x[4 * i + j]) ^ sgn) & 0x80000000u));
    }
    w[i] = canon_nan4(encode2<SAT>(q[0], q[1], o) | (encode2<SAT>(q[2], q[3], o) << 16));
  }
  ovf += o;
  return make_uint4(w[0], w[1], w[2], w[3]);
}

template <int DT, bool SAT>
__device__ __forceinline__ uint4 quantize16(const Raw16<DT>& r, float sc, float y, uint32_t thr, unsigned& ovf,
                                            unsigned& amax) {
  float x[16];
  const uint32_t gm = unpack16<DT>(r, x);
  amax = max(amax, gm);
  if (gm < thr) return encode16_fast(x, sc, y);
  return encode16_exact<SAT>(x, sc, ovf);
}

template <int DT, bool SAT>
__device__ __forceinline__ uint8_t quantize1(const QArgs& a, long long i, float sc, unsigned& ovf, unsigned& amax) {
  float x;
  if (DT == GAS_DTYPE_BF16) {
    const uint16_t b = reinterpret_cast<const uint16_t*>(a.s)[i];
    x = __uint_as_float(static_cast<uint32_t>(b) << 16);
  } else {
    x = reinterpret_cast<const float*>(a.s)[i];
  }
  amax = max(amax, __float_as_uint(x) & 0x7FFFFFFFu);
  const float t = __fdiv_rn(x, sc);
  const uint32_t sgn = __float_as_uint(sc) & 0x80000000u;
  const float q = __uint_as_float((__float_as_uint(t) & 0x7FFFFFFFu) | ((__float_as_uint(x) ^ sgn) & 0x80000000u));
  unsigned o = 0;
  uint32_t c = encode2<SAT>(q, 0.0f, o) & 0xFFu;
  if ((c & 0x7Fu) == 0x7Fu) c = 0x7Fu;
  ovf += o;
  return static_cast<uint8_t>(c);
}

// Bits of the smallest non-negative float a with RN(a / sc) > 448 (sc a positive normal
// float with a normal reciprocal): |x| below it cannot overflow.  RN(a / sc) is
// non-decreasing in a, so stepping from RN(448 sc) to the boundary is exact.
__device__ __forceinline__ uint32_t overflow_threshold(float sc) {
  float t = 448.0f * sc;
  while (__fdiv_rn(t, sc) > kRmax) t = nextafterf(t, 0.0f);
  while (!(__fdiv_rn(t, sc) > kRmax)) t = nextafterf(t, INFINITY);
  return __float_as_uint(t);
}

// Streaming body of the quantize kernel; accumulates the thread's overflow count and amax.
template <int DT, bool SAT>
__device__ __forceinline__ void quantize_body(const QArgs& a, float sc, unsigned& ovf, unsigned& amax) {
  // Groups of sixteen whose largest |x| is below `thr` take the reciprocal path (exact
  // for a positive normal scale with a normal reciprocal); thr = 0 sends every group
  // through the compiler's division.
  const bool fast = sc >= 0x1p-125f && sc <= 0x1p125f;
  const float y = fast ? __frcp_rn(sc) : 0.0f;
  const uint32_t thr = fast ? overflow_threshold(sc) : 0u;
  const long long groups = a.n >> 4;
  const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
  const long long gt = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  long long g = gt;
  // U groups in flight per thread: all loads issued before any group is encoded
  constexpr int U = DT == GAS_DTYPE_BF16 ? 4 : 2;
  for (; g + (U - 1) * stride < groups; g += U * stride) {
    Raw16<DT> r[U];
#pragma unroll
    for (int u = 0; u < U; ++u) load16<DT>(a, g + u * stride, r[u]);
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint4 c = quantize16<DT, SAT>(r[u], sc, y, thr, ovf, amax);
      if (a.q) __stcs(reinterpret_cast<uint4*>(a.q) + g + u * stride, c);
    }
  }
  for (; g < groups; g += stride) {
    Raw16<DT> r;
    load16<DT>(a, g, r);
    const uint4 c = quantize16<DT, SAT>(r, sc, y, thr, ovf, amax);
    if (a.q) __stcs(reinterpret_cast<uint4*>(a.q) + g, c);
  }
  // ragged tail: the last n % 16 logits, one per thread of the first CTA
  const long long i = (groups << 4) + gt;
  if (i < a.n) {
    const uint8_t c = quantize1<DT, SAT>(a, i, sc, ovf, amax);
    if (a.q) a.q[i] = c;
  }
}

template <int DT, bool SAT>
__global__ void __launch_bounds__(kThreads, 3) fp8_quantize_kernel(const __grid_constant__ QArgs a) {
  const float sc = *a.scale;
  unsigned ovf = 0, amax = 0;
  quantize_body<DT, SAT>(a, sc, ovf, amax);

  // CTA reduction -> per-layer accumulator
  __shared__ unsigned s_amax[kThreads / 32];
  __shared__ unsigned s_ovf[kThreads / 32];
  __shared__ bool s_last;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) {
    amax = max(amax, __shfl_xor_sync(0xFFFFFFFFu, amax, off));
    ovf += __shfl_xor_sync(0xFFFFFFFFu, ovf, off);
  }
  if (lane == 0) { s_amax[warp] = amax; s_ovf[warp] = ovf; }
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned m = 0;
    unsigned long long o = 0;
    for (int w = 0; w < kThreads / 32; ++w) { m = max(m, s_amax[w]); o += s_ovf[w]; }
    if (m != 0) atomicMax(&a.acc->amax_bits, m);
    if (o != 0) atomicAdd(&a.acc->overflow, o);
    __threadfence();
    const unsigned t = atomicAdd(&a.acc->ticket, 1u);
    s_last = (t == gridDim.x - 1);
  }
  __syncthreads();
  if (s_last && threadIdx.x == 0) {
    // every other CTA has published its atomics before taking its ticket
    __threadfence();
    const unsigned m = atomicAdd(&a.acc->amax_bits, 0u);
    const unsigned long long o = atomicAdd(&a.acc->overflow, 0ull);
    const float am = __uint_as_float(m);
    gas_fp8_stats st;
    st.amax = am;
    st.max_scaled = __fdiv_rn(am, sc);
    st.overflow = o;
    st.count = static_cast<unsigned long long>(a.n);
    *a.stats = st;
    atomicMax(a.step_amax, m);
    a.acc->amax_bits = 0u;
    a.acc->overflow = 0ull;
    a.acc->ticket = 0u;
  }
}

// NaN-propagating max.
__device__ __forceinline__ float nmax(float m, float v) { return (v > m || v != v) ? v : m; }

__global__ void fp8_delayed_kernel(const float* hist, int layers, int H, float den, float* out) {
  const int l = blockIdx.x * blockDim.x + threadIdx.x;
  if (l >= layers) return;
  float m = hist[static_cast<size_t>(l) * H];
  for (int j = 1; j < H; ++j) m = nmax(m, hist[static_cast<size_t>(l) * H + j]);
  out[l] = __fdiv_rn(m, den);
}

// state[0] = ring position, state[1] = slack steps recorded
__global__ void fp8_end_step_kernel(float* hist, unsigned* step_amax, int* state, int layers, int H,
                                    const float* sigma, int n_q, float c, float* slack, int cap_steps) {
  const int pos = state[0], nrec = state[1];
  for (int l = threadIdx.x; l < layers; l += blockDim.x) {
    const float am = __uint_as_float(step_amax[l]);
    hist[static_cast<size_t>(l) * H + pos] = am;
    step_amax[l] = 0u;
    if (sigma != nullptr && nrec < cap_steps) {
      float sl = sigma[static_cast<size_t>(l) * n_q];
      for (int h = 1; h < n_q; ++h) sl = nmax(sl, sigma[static_cast<size_t>(l) * n_q + h]);
      const float b = sl * c;
      slack[static_cast<size_t>(nrec) * layers + l] = __fdiv_rn(am, b);
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    state[0] = (pos + 1) % H;
    if (sigma != nullptr && nrec < cap_steps) state[1] = nrec + 1;
  }
}

__global__ void fp8_reset_kernel(float* hist, int nh, float init, unsigned* step_amax, LayerAcc* acc, int layers,
                                 int* state) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < nh) hist[i] = init;
  if (i < layers) {
    step_amax[i] = 0u;
    acc[i].amax_bits = 0u;
    acc[i].ticket = 0u;
    acc[i].overflow = 0ull;
  }
  if (i == 0) { state[0] = 0; state[1] = 0; }
}

constexpr int kAlphaThreads = 1024;

__global__ void __launch_bounds__(kAlphaThreads) fp8_auto_alpha_kernel(const float* slack, const int* state,
                                                                        int layers, double q, double kappa,
                                                                        float* alpha_out) {
  extern __shared__ float v[];
  __shared__ int cnt;
  const int total = state[1] * layers;
  if (threadIdx.x == 0) cnt = 0;
  __syncthreads();
  for (int i = threadIdx.x; i < total; i += blockDim.x) {
    const float r = slack[i];
    if (isfinite(r)) v[atomicAdd(&cnt, 1)] = r;
  }
  __syncthreads();
  const int m = cnt;
  int P = 1;
  while (P < m) P <<= 1;
  for (int i = m + threadIdx.x; i < P; i += blockDim.x) v[i] = INFINITY;
  __syncthreads();
  // bitonic sort, ascending
  for (int k = 2; k <= P; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < P; i += blockDim.x) {
        const int p = i ^ j;
        if (p > i) {
          const bool up = (i & k) == 0;
          const float a = v[i], b = v[p];
          if ((a > b) == up) { v[i] = b; v[p] = a; }
        }
      }
      __syncthreads();
    }
  }
  if (threadIdx.x == 0) {
    if (m == 0) {
      *alpha_out = __int_as_float(0x7FC00000);
    } else {
      const double pos = q * static_cast<double>(m - 1);
      int lo = static_cast<int>(floor(pos));
      if (lo > m - 1) lo = m - 1;
      const int hi = lo + 1 < m ? lo + 1 : m - 1;
      const double frac = pos - lo;
      const double x0 = v[lo], x1 = v[hi];
      *alpha_out = static_cast<float>((x0 + frac * (x1 - x0)) * kappa);
    }
  }
}

// Resident CTAs per SM of one kernel instance (queried once).
template <int DT, bool SAT>
int resident_ctas() {
  static int n = 0;
  if (n == 0) {
    int v = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, fp8_quantize_kernel<DT, SAT>, kThreads, 0) != cudaSuccess ||
        v < 1)
      v = 1;
    n = v;
  }
  return n;
}

// One wave of resident CTAs (grid-stride inside), fewer when the input is small.
template <int DT, bool SAT>
cudaError_t launch_quantize(const QArgs& a, int num_sms, cudaStream_t st) {
  const long long groups = a.n >> 4;
  const long long want = (groups + 2LL * kThreads - 1) / (2LL * kThreads);
  const long long cap = static_cast<long long>(num_sms) * resident_ctas<DT, SAT>();
  long long grid = want < cap ? want : cap;
  if (grid < 1) grid = 1;
  fp8_quantize_kernel<DT, SAT><<<static_cast<int>(grid), kThreads, 0, st>>>(a);
  return cudaGetLastError();
}

template <int DT>
cudaError_t launch_quantize_dt(const QArgs& a, bool sat, int num_sms, cudaStream_t st) {
  return sat ? launch_quantize<DT, true>(a, num_sms, st) : launch_quantize<DT, false>(a, num_sms, st);
}

thread_local std::string g_fp8_create_err;

}  // namespace

struct gas_fp8_ctx {
  int layers = 0, H = 0, cap_steps = 0;
  int device = 0, num_sms = 0;
  std::string err;
  void* mem = nullptr;
  float* hist = nullptr;       // [layers][H]
  unsigned* step_amax = nullptr;  // [layers]
  LayerAcc* acc = nullptr;     // [layers]
  int* state = nullptr;        // [2]: ring position, slack steps recorded
  float* slack = nullptr;      // [cap_steps][layers]
};

namespace {

gas_status fp8_fail(gas_fp8_ctx* h, gas_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  if (h) h->err = buf;
  else g_fp8_create_err = buf;
  return st;
}

gas_status fp8_cuda(gas_fp8_ctx* h, cudaError_t e, const char* what) {
  return fp8_fail(h, GAS_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

size_t a256(size_t x) { return (x + 255) / 256 * 256; }
bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace

extern "C" {

gas_status gas_fp8_create(int layers, int history_len, int burn_in_steps, gas_fp8_handle* out) {
  if (out == nullptr) return fp8_fail(nullptr, GAS_ERR_INVALID_ARG, "gas_fp8_create: out is NULL");
  *out = nullptr;
  if (layers < 1 || history_len < 1 || burn_in_steps < 0)
    return fp8_fail(nullptr, GAS_ERR_INVALID_ARG, "gas_fp8_create: layers and history_len must be >= 1, burn_in_steps >= 0");
  if (layers > gas::kMaxLayers || history_len > 1024)
    return fp8_fail(nullptr, GAS_ERR_UNSUPPORTED, "gas_fp8_create: at most %d layers and 1024 history entries",
                    gas::kMaxLayers);
  if (static_cast<long long>(burn_in_steps) * layers > GAS_FP8_MAX_SLACK)
    return fp8_fail(nullptr, GAS_ERR_UNSUPPORTED, "gas_fp8_create: burn_in_steps * layers must be <= %d",
                    GAS_FP8_MAX_SLACK);
  gas_fp8_ctx* h = new (std::nothrow) gas_fp8_ctx();
  if (!h) return fp8_fail(nullptr, GAS_ERR_ALLOC, "gas_fp8_create: out of host memory");
  h->layers = layers;
  h->H = history_len;
  h->cap_steps = burn_in_steps;
  cudaError_t e = cudaGetDevice(&h->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device);
  if (e != cudaSuccess) {
    delete h;
    return fp8_fail(nullptr, GAS_ERR_CUDA, "gas_fp8_create: no usable CUDA device: %s", cudaGetErrorString(e));
  }
  const size_t b_hist = a256(sizeof(float) * layers * history_len);
  const size_t b_step = a256(sizeof(unsigned) * layers);
  const size_t b_acc = a256(sizeof(LayerAcc) * layers);
  const size_t b_state = 256;
  const size_t b_slack = a256(sizeof(float) * (static_cast<size_t>(burn_in_steps) * layers + 1));
  const size_t total = b_hist + b_step + b_acc + b_state + b_slack;
  e = cudaMalloc(&h->mem, total);
  if (e != cudaSuccess) {
    delete h;
    return fp8_fail(nullptr, GAS_ERR_ALLOC, "gas_fp8_create: cudaMalloc(%zu) failed: %s", total, cudaGetErrorString(e));
  }
  char* p = static_cast<char*>(h->mem);
  h->hist = reinterpret_cast<float*>(p); p += b_hist;
  h->step_amax = reinterpret_cast<unsigned*>(p); p += b_step;
  h->acc = reinterpret_cast<LayerAcc*>(p); p += b_acc;
  h->state = reinterpret_cast<int*>(p); p += b_state;
  h->slack = reinterpret_cast<float*>(p);
  e = cudaMemset(h->mem, 0, total);
  if (e == cudaSuccess) {
    const int nh = layers * history_len;
    const int n = nh > layers ? nh : layers;
    fp8_reset_kernel<<<(n + 255) / 256, 256>>>(h->hist, nh, 1.0f, h->step_amax, h->acc, layers, h->state);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    cudaFree(h->mem);
    delete h;
    return fp8_fail(nullptr, GAS_ERR_CUDA, "gas_fp8_create: initialisation failed: %s", cudaGetErrorString(e));
  }
  *out = h;
  return GAS_OK;
}

gas_status gas_fp8_destroy(gas_fp8_handle h) {
  if (!h) return GAS_ERR_INVALID_ARG;
  cudaFree(h->mem);
  delete h;
  return GAS_OK;
}

gas_status gas_fp8_reset(gas_fp8_handle h, float history_init, void* stream) {
  if (!h) return GAS_ERR_INVALID_ARG;
  const int nh = h->layers * h->H;
  const int n = nh > h->layers ? nh : h->layers;
  fp8_reset_kernel<<<(n + 255) / 256, 256, 0, static_cast<cudaStream_t>(stream)>>>(
      h->hist, nh, history_init, h->step_amax, h->acc, h->layers, h->state);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? GAS_OK : fp8_cuda(h, e, "gas_fp8_reset");
}

gas_status gas_fp8_delayed_scales(gas_fp8_handle h, double eta, float* scale_out, void* stream) {
  if (!h) return GAS_ERR_INVALID_ARG;
  if (!(eta > 0.0)) return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_delayed_scales: eta must be > 0");
  if (!scale_out || !aligned(scale_out, 4))
    return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_delayed_scales: scale_out NULL or misaligned");
  const float den = static_cast<float>(448.0 * eta);
  fp8_delayed_kernel<<<(h->layers + 127) / 128, 128, 0, static_cast<cudaStream_t>(stream)>>>(h->hist, h->layers,
                                                                                           h->H, den, scale_out);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? GAS_OK : fp8_cuda(h, e, "gas_fp8_delayed_scales");
}

gas_status gas_fp8_quantize(gas_fp8_handle h, int layer, const void* s, int dtype, long long n, const float* scale,
                            unsigned char* q_out, int flags, gas_fp8_stats* stats, void* stream) {
  if (!h) return GAS_ERR_INVALID_ARG;
  if (layer < 0 || layer >= h->layers)
    return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_quantize: layer %d outside [0, %d)", layer, h->layers);
  if (n < 0) return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_quantize: n must be >= 0");
  if (dtype != GAS_DTYPE_BF16 && dtype != GAS_DTYPE_F32)
    return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_quantize: unknown dtype %d", dtype);
  if (!scale || !aligned(scale, 4)) return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_quantize: scale NULL or misaligned");
  if (!stats || !aligned(stats, 8)) return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_quantize: stats NULL or misaligned");
  if (n > 0 && (!s || !aligned(s, 16)))
    return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_quantize: logits NULL or not 16-byte aligned");
  if (q_out && !aligned(q_out, 16))
    return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_quantize: q_out not 16-byte aligned");
  if (flags & ~GAS_FP8_SATURATE) return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_quantize: unknown flags 0x%x", flags);
  QArgs a{};
  a.s = s;
  a.n = n;
  a.scale = scale;
  a.q = q_out;
  a.acc = h->acc + layer;
  a.step_amax = h->step_amax + layer;
  a.stats = stats;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const bool sat = (flags & GAS_FP8_SATURATE) != 0;
  cudaError_t e;
  if (dtype == GAS_DTYPE_BF16) e = launch_quantize_dt<GAS_DTYPE_BF16>(a, sat, h->num_sms, st);
  else e = launch_quantize_dt<GAS_DTYPE_F32>(a, sat, h->num_sms, st);
  return e == cudaSuccess ? GAS_OK : fp8_cuda(h, e, "gas_fp8_quantize");
}

gas_status gas_fp8_end_step(gas_fp8_handle h, const float* sigma, int n_q, int d, int d_h, void* stream) {
  if (!h) return GAS_ERR_INVALID_ARG;
  if (sigma && (n_q < 1 || d < 1 || d_h < 1))
    return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_end_step: n_q, d and d_h must be >= 1");
  if (sigma && !aligned(sigma, 4)) return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_end_step: sigma misaligned");
  const float c = sigma ? static_cast<float>(static_cast<double>(d) / std::sqrt(static_cast<double>(d_h))) : 0.0f;
  const int threads = h->layers < 1024 ? ((h->layers + 31) / 32) * 32 : 1024;
  fp8_end_step_kernel<<<1, threads, 0, static_cast<cudaStream_t>(stream)>>>(
      h->hist, h->step_amax, h->state, h->layers, h->H, sigma, n_q, c, h->slack, h->cap_steps);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? GAS_OK : fp8_cuda(h, e, "gas_fp8_end_step");
}

gas_status gas_fp8_auto_alpha(gas_fp8_handle h, double q, double kappa, float* alpha_out, void* stream) {
  if (!h) return GAS_ERR_INVALID_ARG;
  if (!(q >= 0.0 && q <= 1.0)) return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_auto_alpha: q must be in [0, 1]");
  if (!(kappa > 0.0)) return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_auto_alpha: kappa must be > 0");
  if (!alpha_out || !aligned(alpha_out, 4))
    return fp8_fail(h, GAS_ERR_INVALID_ARG, "gas_fp8_auto_alpha: alpha_out NULL or misaligned");
  int P = 1;
  while (P < h->cap_steps * h->layers) P <<= 1;
  const size_t smem = sizeof(float) * static_cast<size_t>(P);
  cudaError_t e = cudaSuccess;
  if (smem > 48 * 1024)
    e = cudaFuncSetAttribute(fp8_auto_alpha_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e == cudaSuccess) {
    fp8_auto_alpha_kernel<<<1, kAlphaThreads, smem, static_cast<cudaStream_t>(stream)>>>(h->slack, h->state, h->layers,
                                                                                         q, kappa, alpha_out);
    e = cudaGetLastError();
  }
  return e == cudaSuccess ? GAS_OK : fp8_cuda(h, e, "gas_fp8_auto_alpha");
}

gas_status gas_fp8_slack_count(gas_fp8_handle h, int* count) {
  if (!h || !count) return GAS_ERR_INVALID_ARG;
  int st[2] = {0, 0};
  const cudaError_t e = cudaMemcpy(st, h->state, sizeof(st), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fp8_cuda(h, e, "gas_fp8_slack_count");
  *count = st[1] * h->layers;
  return GAS_OK;
}

const char* gas_fp8_last_error(gas_fp8_handle h) { return h ? h->err.c_str() : g_fp8_create_err.c_str(); }

}  // extern "C"
