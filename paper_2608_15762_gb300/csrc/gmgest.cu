// Online linear estimators (Sec. 3.3.1): batched least-squares refits from
// executor feedback and the integer duration / link tables they produce for
// the simulation.  The C ABI is declared in include/gmgest.h.
//
// est_update, in three launches:
//  1. chunk counts: every estimator's samples are cut into chunks of kChunk
//     rows; one block computes the exclusive prefix of the chunk counts;
//  2. one warp per chunk: lane l sums rows l, l+32, ... of the chunk into the
//     upper triangle of X^T X, X^T y and a count (fp64), the 32 partial sums
//     are combined by a fixed shfl_xor tree and written to the caller's
//     buffer -- enough independent loads in flight to stream the samples at
//     memory speed;
//  3. one warp per estimator: lane l adds the partials of chunks l, l+32, ...,
//     a fixed shfl_xor tree combines the lanes, lane 0 adds the result to the
//     running statistics and refits by a Cholesky solve of the normal
//     equations.
// Every sum has a fixed order, so results do not depend on scheduling.  F
// (<= 8) is a template parameter so the per-sample arrays stay in registers.

#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "../../include/gmgest.h"

namespace gest {
namespace {

constexpr unsigned kFullMask = 0xffffffffu;
constexpr double kPivotRel = 1e-12;   // pivot threshold relative to its own diagonal entry
constexpr int64_t kMaxTicks = int64_t(1) << 40;
constexpr int32_t kChunk = 128;       // sample rows per warp in the first reduction pass

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// State layout (each array 256-byte aligned): G [E][F(F+1)/2] upper triangle
// row-major, h [E][F], n [E], beta [E][F], fitted [E] (int32).
struct Layout {
  size_t g, h, n, beta, fitted, total;
};

Layout layout(int32_t E, int32_t F) {
  Layout L;
  const size_t tri = (size_t)F * (F + 1) / 2;
  size_t o = 0;
  L.g = o;
  o = align256(o + 8 * tri * (size_t)E);
  L.h = o;
  o = align256(o + 8 * (size_t)F * E);
  L.n = o;
  o = align256(o + 8 * (size_t)E);
  L.beta = o;
  o = align256(o + 8 * (size_t)F * E);
  L.fitted = o;
  o = align256(o + 4 * (size_t)E);
  L.total = o;
  return L;
}

struct State {
  double* g;
  double* h;
  double* n;
  double* beta;
  int32_t* fitted;
};

State view(void* d_state, int32_t E, int32_t F) {
  const Layout L = layout(E, F);
  uint8_t* b = static_cast<uint8_t*>(d_state);
  return State{reinterpret_cast<double*>(b + L.g), reinterpret_cast<double*>(b + L.h),
               reinterpret_cast<double*>(b + L.n), reinterpret_cast<double*>(b + L.beta),
               reinterpret_cast<int32_t*>(b + L.fitted)};
}

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFullMask, v, o);
  return v;
}

// Chunk prefix: chunks[e] = exclusive prefix of ceil(count_e / kChunk);
// chunks[E] = total.  One block; thread t takes a contiguous run of
// estimators.
__global__ void __launch_bounds__(1024) est_chunks_kernel(int32_t E, const int32_t* __restrict__ off,
                                                          int32_t* __restrict__ chunks) {
  __shared__ int32_t part[1024];
  const int t = threadIdx.x;
  const int32_t per = (E + 1023) / 1024;
  const int32_t e0 = min(E, t * per), e1 = min(E, e0 + per);
  int32_t sum = 0;
  for (int32_t e = e0; e < e1; ++e) sum += (off[e + 1] - off[e] + kChunk - 1) / kChunk;
  part[t] = sum;
  __syncthreads();
  for (int o = 1; o < 1024; o <<= 1) {  // inclusive scan (Hillis-Steele)
    const int32_t v = t >= o ? part[t - o] : 0;
    __syncthreads();
    part[t] += v;
    __syncthreads();
  }
  int32_t acc = part[t] - sum;
  for (int32_t e = e0; e < e1; ++e) {
    chunks[e] = acc;
    acc += (off[e + 1] - off[e] + kChunk - 1) / kChunk;
  }
  if (t == 1023) chunks[E] = part[1023];
}

// One warp per chunk: partial statistics [T triangle | F | count].
template <int F>
__global__ void __launch_bounds__(128) est_partial_kernel(int32_t E, int64_t max_chunks,
                                                          const int32_t* __restrict__ off,
                                                          const int32_t* __restrict__ chunks,
                                                          const double* __restrict__ x,
                                                          const double* __restrict__ y,
                                                          double* __restrict__ partial) {
  constexpr int T = F * (F + 1) / 2;
  constexpr int P = T + F + 1;
  const int lane = threadIdx.x & 31;
  const int64_t c = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (c >= max_chunks || c >= chunks[E]) return;  // whole warps leave together
  // the estimator whose chunk range holds c: the last e with chunks[e] <= c
  int32_t lo = 0, hi = E - 1;
  while (lo < hi) {
    const int32_t mid = (lo + hi + 1) >> 1;
    if (chunks[mid] <= c) lo = mid;
    else hi = mid - 1;
  }
  const int32_t e = lo;
  const int32_t r0 = off[e] + (int32_t)(c - chunks[e]) * kChunk;
  const int32_t r1 = min(off[e + 1], r0 + kChunk);
  double g[T], h[F], cnt = 0.0;
#pragma unroll
  for (int t = 0; t < T; ++t) g[t] = 0.0;
#pragma unroll
  for (int a = 0; a < F; ++a) h[a] = 0.0;
  // rows r and r + 32 per step: twice the loads in flight, same summation
  // order for every run
  for (int32_t r = r0 + lane; r < r1; r += 64) {
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int32_t rr = r + 32 * half;
      if (rr < r1) {
        double xv[F];
#pragma unroll
        for (int a = 0; a < F; ++a) xv[a] = x[(int64_t)rr * F + a];
        const double yv = y[rr];
        int t = 0;
#pragma unroll
        for (int a = 0; a < F; ++a) {
          h[a] += xv[a] * yv;
#pragma unroll
          for (int b = a; b < F; ++b) g[t++] += xv[a] * xv[b];
        }
        cnt += 1.0;
      }
    }
  }
#pragma unroll
  for (int t = 0; t < T; ++t) g[t] = warp_sum(g[t]);
#pragma unroll
  for (int a = 0; a < F; ++a) h[a] = warp_sum(h[a]);
  cnt = warp_sum(cnt);
  if (lane != 0) return;
  double* out = partial + c * P;
#pragma unroll
  for (int t = 0; t < T; ++t) out[t] = g[t];
#pragma unroll
  for (int a = 0; a < F; ++a) out[T + a] = h[a];
  out[T + F] = cnt;
}

// One warp per estimator: add the chunk partials (fixed order), then refit.
template <int F>
__global__ void __launch_bounds__(128) est_fit_kernel(State S, int32_t E, const int32_t* __restrict__ chunks,
                                                      const double* __restrict__ partial) {
  constexpr int T = F * (F + 1) / 2;
  constexpr int P = T + F + 1;
  const int lane = threadIdx.x & 31;
  const int64_t e = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (e >= E) return;  // whole warps leave together
  double g[T], h[F], cnt = 0.0;
#pragma unroll
  for (int t = 0; t < T; ++t) g[t] = 0.0;
#pragma unroll
  for (int a = 0; a < F; ++a) h[a] = 0.0;
  for (int32_t c = chunks[e] + lane; c < chunks[e + 1]; c += 32) {
    const double* p = partial + (int64_t)c * P;
#pragma unroll
    for (int t = 0; t < T; ++t) g[t] += p[t];
#pragma unroll
    for (int a = 0; a < F; ++a) h[a] += p[T + a];
    cnt += p[T + F];
  }
#pragma unroll
  for (int t = 0; t < T; ++t) g[t] = warp_sum(g[t]);
#pragma unroll
  for (int a = 0; a < F; ++a) h[a] = warp_sum(h[a]);
  cnt = warp_sum(cnt);
  if (lane != 0) return;
  double* G = S.g + e * T;
  double* H = S.h + e * F;
#pragma unroll
  for (int t = 0; t < T; ++t) g[t] = (G[t] += g[t]);
#pragma unroll
  for (int a = 0; a < F; ++a) h[a] = (H[a] += h[a]);
  const double n = (S.n[e] += cnt);
  // Cholesky factor L (lower) of the full matrix built from the triangle
  double A[F][F];
  {
    int t = 0;
#pragma unroll
    for (int a = 0; a < F; ++a)
#pragma unroll
      for (int b = a; b < F; ++b) {
        A[a][b] = g[t];
        A[b][a] = g[t];
        ++t;
      }
  }
  // A pivot is compared with its own diagonal entry, which makes the test
  // independent of each feature's scale (bytes next to a constant term).
  bool ok = n >= (double)F;
  double L[F][F];
#pragma unroll
  for (int j = 0; j < F; ++j) {
    double d = A[j][j];
#pragma unroll
    for (int k = 0; k < j; ++k) d -= L[j][k] * L[j][k];
    ok = ok && d > kPivotRel * A[j][j];
    const double ljj = sqrt(fmax(d, 0.0));
    L[j][j] = ljj;
#pragma unroll
    for (int i = j + 1; i < F; ++i) {
      double v = A[i][j];
#pragma unroll
      for (int k = 0; k < j; ++k) v -= L[i][k] * L[j][k];
      L[i][j] = ok ? v / ljj : 0.0;
    }
  }
  double beta[F];
  if (ok) {
    double z[F];
#pragma unroll
    for (int i = 0; i < F; ++i) {
      double v = h[i];
#pragma unroll
      for (int k = 0; k < i; ++k) v -= L[i][k] * z[k];
      z[i] = v / L[i][i];
    }
#pragma unroll
    for (int i = F - 1; i >= 0; --i) {
      double v = z[i];
#pragma unroll
      for (int k = i + 1; k < F; ++k) v -= L[k][i] * beta[k];
      beta[i] = v / L[i][i];
    }
  } else {
#pragma unroll
    for (int i = 0; i < F; ++i) beta[i] = 0.0;
  }
#pragma unroll
  for (int a = 0; a < F; ++a) S.beta[e * F + a] = beta[a];
  S.fitted[e] = ok ? 1 : 0;
}

__device__ __forceinline__ int64_t clamp_rint(double v, int64_t lo) {
  const double r = rint(v);
  if (!(r >= (double)lo)) return lo;  // also NaN
  if (r >= (double)kMaxTicks) return kMaxTicks;
  return (int64_t)r;
}

__global__ void __launch_bounds__(256) est_predict_kernel(State S, int32_t F, int64_t NT, int32_t T,
                                                          const int32_t* __restrict__ est_of,
                                                          const double* __restrict__ x,
                                                          const int64_t* __restrict__ dflt,
                                                          int64_t* __restrict__ dur) {
  const int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (q >= NT) return;
  const int64_t i = q / T;
  const int32_t e = est_of[q];
  if (e < 0 || !S.fitted[e]) {
    dur[q] = dflt[i];
    return;
  }
  double v = 0.0;
  for (int a = 0; a < F; ++a) v += S.beta[(int64_t)e * F + a] * x[i * F + a];
  dur[q] = clamp_rint(v, 1);
}

__global__ void __launch_bounds__(256) est_links_kernel(State S, int32_t D, const int64_t* __restrict__ bw_dflt,
                                                        const int64_t* __restrict__ lat_dflt,
                                                        int64_t* __restrict__ bw, int64_t* __restrict__ lat) {
  const int32_t q = blockIdx.x * blockDim.x + threadIdx.x;
  if (q >= D * D) return;
  const int32_t d = q / D, e = q % D;
  if (d == e || !S.fitted[q]) {
    bw[q] = bw_dflt[q];
    lat[q] = lat_dflt[q];
    return;
  }
  const double alpha = S.beta[2 * (int64_t)q], c = S.beta[2 * (int64_t)q + 1];
  bw[q] = alpha > 0.0 ? clamp_rint(1.0 / alpha, 1) : kMaxTicks;
  lat[q] = clamp_rint(c, 0);
}

// Upper bound of the chunk count: sum over e of ceil(count_e / kChunk).
int64_t max_chunks(int32_t E, int64_t S) { return S / kChunk + E; }

template <int F>
cudaError_t launch_update(State S, int32_t E, int64_t nsamp, const int32_t* off, const double* x,
                          const double* y, int32_t* chunks, double* partial, cudaStream_t st) {
  const int64_t mc = max_chunks(E, nsamp);
  est_chunks_kernel<<<1, 1024, 0, st>>>(E, off, chunks);
  if (mc > 0) est_partial_kernel<F><<<(int)((mc * 32 + 127) / 128), 128, 0, st>>>(E, mc, off, chunks, x, y, partial);
  est_fit_kernel<F><<<(int)(((int64_t)E * 32 + 127) / 128), 128, 0, st>>>(S, E, chunks, partial);
  return cudaGetLastError();
}

// Caller buffer of est_update: chunk prefix [E+1] int32, then the partials
// [max chunks][F(F+1)/2 + F + 1] fp64.
size_t tmp_partial_off(int32_t E) { return align256(4 * ((size_t)E + 1)); }
size_t tmp_bytes(int32_t E, int32_t F, int64_t S) {
  const size_t P = (size_t)F * (F + 1) / 2 + F + 1;
  return tmp_partial_off(E) + align256(8 * P * (size_t)max_chunks(E, S));
}

bool args_ok(const void* state, int32_t E, int32_t F) {
  return state && E >= 1 && F >= 1 && F <= GMG_EST_MAX_FEATURES &&
         (reinterpret_cast<uintptr_t>(state) & 255) == 0;
}

}  // namespace
}  // namespace gest

using namespace gest;

extern "C" {

size_t est_state_bytes(int32_t n_est, int32_t n_feat) {
  if (n_est < 1 || n_feat < 1 || n_feat > GMG_EST_MAX_FEATURES) return 0;
  return layout(n_est, n_feat).total;
}

int est_reset(void* d_state, int32_t n_est, int32_t n_feat, gmg_stream_t stream) {
  if (!args_ok(d_state, n_est, n_feat)) return GMG_EINVAL;
  const cudaError_t e =
      cudaMemsetAsync(d_state, 0, layout(n_est, n_feat).total, reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? GMG_OK : GMG_ECUDA;
}

size_t est_update_tmp_bytes(int32_t n_est, int32_t n_feat, int64_t n_samples) {
  if (n_est < 1 || n_feat < 1 || n_feat > GMG_EST_MAX_FEATURES || n_samples < 0) return 0;
  return tmp_bytes(n_est, n_feat, n_samples);
}

int est_update(void* d_state, int32_t n_est, int32_t n_feat, const int32_t* d_off, const double* d_x,
               const double* d_y, int64_t n_samples, void* d_tmp, size_t tmp_bytes_given, gmg_stream_t stream) {
  if (!args_ok(d_state, n_est, n_feat) || !d_off || n_samples < 0 || n_samples > INT32_MAX) return GMG_EINVAL;
  if (n_samples > 0 && (!d_x || !d_y)) return GMG_EINVAL;
  if (!d_tmp || (reinterpret_cast<uintptr_t>(d_tmp) & 255) != 0 ||
      tmp_bytes_given < tmp_bytes(n_est, n_feat, n_samples))
    return GMG_EWS;
  const State S = view(d_state, n_est, n_feat);
  const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int32_t* chunks = static_cast<int32_t*>(d_tmp);
  double* partial = reinterpret_cast<double*>(static_cast<uint8_t*>(d_tmp) + tmp_partial_off(n_est));
  cudaError_t e = cudaSuccess;
  switch (n_feat) {
    case 1: e = launch_update<1>(S, n_est, n_samples, d_off, d_x, d_y, chunks, partial, st); break;
    case 2: e = launch_update<2>(S, n_est, n_samples, d_off, d_x, d_y, chunks, partial, st); break;
    case 3: e = launch_update<3>(S, n_est, n_samples, d_off, d_x, d_y, chunks, partial, st); break;
    case 4: e = launch_update<4>(S, n_est, n_samples, d_off, d_x, d_y, chunks, partial, st); break;
    case 5: e = launch_update<5>(S, n_est, n_samples, d_off, d_x, d_y, chunks, partial, st); break;
    case 6: e = launch_update<6>(S, n_est, n_samples, d_off, d_x, d_y, chunks, partial, st); break;
    case 7: e = launch_update<7>(S, n_est, n_samples, d_off, d_x, d_y, chunks, partial, st); break;
    default: e = launch_update<8>(S, n_est, n_samples, d_off, d_x, d_y, chunks, partial, st); break;
  }
  return e == cudaSuccess ? GMG_OK : GMG_ECUDA;
}

int est_coefficients(const void* d_state, int32_t n_est, int32_t n_feat, double* d_beta, int32_t* d_fitted,
                     gmg_stream_t stream) {
  if (!args_ok(d_state, n_est, n_feat)) return GMG_EINVAL;
  const State S = view(const_cast<void*>(d_state), n_est, n_feat);
  const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (d_beta && cudaMemcpyAsync(d_beta, S.beta, 8 * (size_t)n_est * n_feat, cudaMemcpyDeviceToDevice, st) !=
                    cudaSuccess)
    return GMG_ECUDA;
  if (d_fitted &&
      cudaMemcpyAsync(d_fitted, S.fitted, 4 * (size_t)n_est, cudaMemcpyDeviceToDevice, st) != cudaSuccess)
    return GMG_ECUDA;
  return GMG_OK;
}

int est_predict_durations(const void* d_state, int32_t n_est, int32_t n_feat, int32_t n_ops, int32_t n_types,
                          const int32_t* d_est_of, const double* d_x, const int64_t* d_dflt, int64_t* d_dur,
                          gmg_stream_t stream) {
  if (!args_ok(d_state, n_est, n_feat) || n_ops < 0 || n_types < 1) return GMG_EINVAL;
  const int64_t NT = (int64_t)n_ops * n_types;
  if (NT == 0) return GMG_OK;
  if (!d_est_of || !d_x || !d_dflt || !d_dur) return GMG_EINVAL;
  const State S = view(const_cast<void*>(d_state), n_est, n_feat);
  const int blocks = (int)((NT + 255) / 256);
  est_predict_kernel<<<blocks, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(S, n_feat, NT, n_types,
                                                                                  d_est_of, d_x, d_dflt, d_dur);
  return cudaGetLastError() == cudaSuccess ? GMG_OK : GMG_ECUDA;
}

int est_links(const void* d_state, int32_t n_dev, const int64_t* d_bw_dflt, const int64_t* d_lat_dflt,
              int64_t* d_bw, int64_t* d_lat, gmg_stream_t stream) {
  if (n_dev < 1 || n_dev > 256 || !args_ok(d_state, n_dev * n_dev, 2)) return GMG_EINVAL;
  if (!d_bw_dflt || !d_lat_dflt || !d_bw || !d_lat) return GMG_EINVAL;
  const State S = view(const_cast<void*>(d_state), n_dev * n_dev, 2);
  const int n = n_dev * n_dev;
  est_links_kernel<<<(n + 255) / 256, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(S, n_dev, d_bw_dflt,
                                                                                          d_lat_dflt, d_bw, d_lat);
  return cudaGetLastError() == cudaSuccess ? GMG_OK : GMG_ECUDA;
}

}  // extern "C"
