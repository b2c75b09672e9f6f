// Per-call batch kernels of the scoring path: ragged packing and ranking.
//
// pack: builds the decoder input X = [candidate rows of all requests; context
// rows of all requests] (App. B token sequence, per request [ctx; cand]),
// the row -> request map used by the attention kernels, and the part of the
// action logits that depends only on the raw candidate token x
// (Sec. 4.1.3 with linear f_dec: logits = z Weff_z + x Weff_x + b_dec Q_dec^T).
// The host passes the candidate offsets by value (no host->device copy).
//
// rank: per request, candidate indices by descending probability of one
// action, ties to the lower index, NaN last (an exact counting rank).
#include "txs_internal.cuh"

namespace txs {

constexpr int kMaxReqParamV = 4096;
extern const int kMaxReqParam = kMaxReqParamV;

struct PackArgs {
  int n_req, n_cand, S, d, na;
  int cand_off[kMaxReqParamV + 1];
};

struct RankArgs {
  int n_req, na, action, top_k;
  int cand_off[kMaxReqParamV + 1];
};

namespace {

__device__ __forceinline__ int find_segment_param(const int* off, int n, int row) {
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (off[mid] <= row) lo = mid; else hi = mid - 1;
  }
  return lo;
}

constexpr int kPackRowsPerWarp = 4;

// Sum of NA per-lane values over the 32 lanes of a warp, scattered: on return
// every lane holds the total of value lane / (32 / NA).  Each halving step
// exchanges half of the remaining values with the partner lane (NA - 1
// shuffles in all), then the lanes that share a value finish with a butterfly.
template <int NA>
__device__ __forceinline__ float warp_reduce_scatter(float (&v)[NA], int lane) {
#pragma unroll
  for (int h = NA / 2, o = 16; h >= 1; h >>= 1, o >>= 1) {
    const bool upper = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < h; ++i) {
      const float send = upper ? v[i] : v[i + h];
      const float keep = upper ? v[i + h] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
    }
  }
  float x = v[0];
#pragma unroll
  for (int o = 16 / NA; o >= 1; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// 8 warps per CTA, kPackRowsPerWarp consecutive rows per warp (all of a
// warp's row loads are issued before its arithmetic); CH 16-byte chunks per
// lane and row cover d.  The x-part of the logits takes NA >= na actions (the
// actions na..NA-1 have zero weights and are not written); the head weights
// are staged per CTA in shared memory as [action][column] and read as float4
// runs, which keeps the register count low enough for four CTAs per SM and
// so many rows in flight.
template <typename T, int NA, int CH>
__global__ void __launch_bounds__(256) pack_kernel(const __grid_constant__ PackArgs a, const T* __restrict__ cand,
                                                   const T* __restrict__ ctx, T* __restrict__ X,
                                                   int* __restrict__ row_req, int* __restrict__ cand_off_dev,
                                                   const float* __restrict__ weff_x,
                                                   const float* __restrict__ cdec, float* __restrict__ xlog) {
  pdl_launch_dependents();
  pdl_wait();
  constexpr int VEC = Vec16<T>::N;
  constexpr int MAXCH = CH;
  extern __shared__ float4 sw4[];
  float* sw = reinterpret_cast<float*>(sw4);    // [NA][d]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int d = a.d, na = a.na;
  if (blockIdx.x == 0)
    for (int i = threadIdx.x; i <= a.n_req; i += 256) cand_off_dev[i] = a.cand_off[i];
  const long long n_rows = a.n_cand + static_cast<long long>(a.n_req) * a.S;
  const long long p0 = (static_cast<long long>(blockIdx.x) * 8 + warp) * kPackRowsPerWarp;
  uint4 raw[kPackRowsPerWarp][MAXCH];
#pragma unroll
  for (int t = 0; t < kPackRowsPerWarp; ++t) {
    const long long p = p0 + t;
    const T* src = p < a.n_cand ? cand + p * d : (p < n_rows ? ctx + (p - a.n_cand) * d : cand);
#pragma unroll
    for (int j = 0; j < MAXCH; ++j) {
      const int col = (j * 32 + lane) * VEC;
      raw[t][j] = (p < n_rows && col < d) ? *reinterpret_cast<const uint4*>(src + col) : make_uint4(0, 0, 0, 0);
    }
  }
  // head weights, staged after the row loads are in flight
  for (int c = threadIdx.x; c < d; c += 256)
#pragma unroll
    for (int k = 0; k < NA; ++k) sw[k * d + c] = k < na ? weff_x[static_cast<long long>(c) * na + k] : 0.f;
  __syncthreads();
#pragma unroll
  for (int t = 0; t < kPackRowsPerWarp; ++t) {
    const long long p = p0 + t;
    if (p >= n_rows) break;                     // uniform over the warp
    const bool is_cand = p < a.n_cand;
    T* dst = X + p * d;
#pragma unroll
    for (int j = 0; j < MAXCH; ++j) {
      const int col = (j * 32 + lane) * VEC;
      if (col < d) *reinterpret_cast<uint4*>(dst + col) = raw[t][j];
    }
    if (lane == 0)
      row_req[p] = is_cand ? find_segment_param(a.cand_off, a.n_req, static_cast<int>(p))
                           : static_cast<int>((p - a.n_cand) / a.S);
    if (is_cand) {
      float lg[NA];
#pragma unroll
      for (int k = 0; k < NA; ++k) lg[k] = 0.f;
#pragma unroll
      for (int j = 0; j < MAXCH; ++j) {
        const int col = (j * 32 + lane) * VEC;
        if (col < d) {
          float v[VEC];
          Vec16<T>::load(reinterpret_cast<const T*>(&raw[t][j]), v);
#pragma unroll
          for (int k = 0; k < NA; ++k) {
            const float4* w4 = reinterpret_cast<const float4*>(sw + k * d + col);
            float acc = 0.f;
#pragma unroll
            for (int qq = 0; qq < VEC / 4; ++qq) {
              const float4 w = w4[qq];
              acc = fmaf(v[4 * qq], w.x, acc);
              acc = fmaf(v[4 * qq + 1], w.y, acc);
              acc = fmaf(v[4 * qq + 2], w.z, acc);
              acc = fmaf(v[4 * qq + 3], w.w, acc);
            }
            lg[k] += acc;
          }
        }
      }
      const float x = warp_reduce_scatter<NA>(lg, lane);
      const int k = lane / (32 / NA);
      if ((lane & (32 / NA - 1)) == 0 && k < na) xlog[p * na + k] = x + __ldg(cdec + k);
    }
  }
}

// Monotone map of a float to uint32 for descending comparison; NaN -> 0
// (after every number), -0 -> +0.
__device__ __forceinline__ uint32_t order_key(float f) {
  if (f != f) return 0u;
  uint32_t u = __float_as_uint(f);
  if ((u & 0x7FFFFFFFu) == 0) u = 0;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__global__ void __launch_bounds__(1024) rank_kernel(const __grid_constant__ RankArgs a, const float* __restrict__ probs,
                                                    int* __restrict__ out) {
  pdl_launch_dependents();
  pdl_wait();
  extern __shared__ uint32_t keys[];
  const int r = blockIdx.x;
  const int c0 = a.cand_off[r];
  const int M = a.cand_off[r + 1] - c0;
  for (int i = threadIdx.x; i < M; i += blockDim.x)
    keys[i] = order_key(probs[static_cast<long long>(c0 + i) * a.na + a.action]);
  __syncthreads();
  // CTA y of the request ranks candidates [i0, i1) against all M keys
  const int per = (M + static_cast<int>(gridDim.y) - 1) / static_cast<int>(gridDim.y);
  const int i0 = static_cast<int>(blockIdx.y) * per;
  const int i1 = min(M, i0 + per);
  const int n_i = i1 > i0 ? i1 - i0 : 0;
  // tpc consecutive lanes share a candidate (short slates leave threads to
  // spare), each counting every tpc-th key with four independent counters;
  // the group adds its counts with shuffles.  Every lane runs the same number
  // of rounds, so the shuffles see full warps.
  int tpc = 1;
  while (tpc < 32 && tpc * 2 * n_i <= static_cast<int>(blockDim.x)) tpc *= 2;
  const int per_round = blockDim.x / tpc;
  const int sub = threadIdx.x & (tpc - 1);
  const int rounds = (n_i + per_round - 1) / per_round;
  for (int round = 0; round < rounds; ++round) {
    const int i = i0 + round * per_round + static_cast<int>(threadIdx.x) / tpc;
    int rank = 0;
    if (i < i1) {
      const uint32_t ki = keys[i];
      int c[4] = {0, 0, 0, 0};
      int j = sub;
      for (; j + 3 * tpc < M; j += 4 * tpc) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int jj = j + u * tpc;
          const uint32_t kj = keys[jj];
          c[u] += (kj > ki) | ((kj == ki) & (jj < i));
        }
      }
      for (; j < M; j += tpc) {
        const uint32_t kj = keys[j];
        c[0] += (kj > ki) | ((kj == ki) & (j < i));
      }
      rank = (c[0] + c[1]) + (c[2] + c[3]);
    }
    for (int o = tpc >> 1; o >= 1; o >>= 1) rank += __shfl_xor_sync(0xffffffffu, rank, o);
    if (i < i1 && sub == 0) {
      if (a.top_k == 0) out[c0 + rank] = i;
      else if (rank < a.top_k) out[static_cast<long long>(r) * a.top_k + rank] = i;
    }
  }
  if (a.top_k > 0 && blockIdx.y == 0)
    for (int t = M + threadIdx.x; t < a.top_k; t += blockDim.x) out[static_cast<long long>(r) * a.top_k + t] = -1;
}

// Small host int arrays reach the device as kernel parameters (copied by
// value at launch: no copy-engine transfer, nothing left behind in host
// memory, so the call can be captured into a CUDA graph).  Two segments, a
// then b, in one launch; it waits for the preceding kernel first, which may
// still be reading the old values.
template <int N>
struct UploadArgs {
  int* dst_a;
  int* dst_b;
  int n_a, n_b;
  int v[N];
};

template <int N>
__global__ void __launch_bounds__(256) upload_kernel(const __grid_constant__ UploadArgs<N> a) {
  pdl_launch_dependents();
  pdl_wait();
  for (int i = blockIdx.x * 256 + threadIdx.x; i < a.n_a + a.n_b; i += gridDim.x * 256) {
    if (i < a.n_a) a.dst_a[i] = a.v[i];
    else a.dst_b[i - a.n_a] = a.v[i];
  }
}

// Deep & Wide head input: row i of Z2 = [z_i, x_i[dw_in:]] for the candidate
// rows (z: the decoder output, x: the raw candidate token).  One warp per row,
// 16-byte vectors.
template <typename T>
__global__ void __launch_bounds__(256) dw_gather_kernel(const T* __restrict__ Z, const T* __restrict__ cand,
                                                        T* __restrict__ Z2, int n_cand, int d, int dw_in) {
  pdl_launch_dependents();
  pdl_wait();
  constexpr int VEC = Vec16<T>::N;
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= n_cand) return;
  const int w2 = 2 * d - dw_in;
  T* dst = Z2 + static_cast<long long>(row) * w2;
  for (int c = lane * VEC; c < w2; c += 32 * VEC) {
    float v[VEC];
    if (c < d) Vec16<T>::load(Z + static_cast<long long>(row) * d + c, v);
    else Vec16<T>::load(cand + static_cast<long long>(row) * d + dw_in + (c - d), v);
    Vec16<T>::store(dst + c, v);
  }
}

// Deep & Wide head output: logits[i] = xlog[i] + h_i w2q, probs = softmax
// (h = GELU([z, x_deep] W_d1 + b_d1), w2q = W_d2 Q_deep^T folded).  One warp
// per candidate row; the fold keeps the Fh x k product in fp32.
template <typename T>
__global__ void __launch_bounds__(256) dw_head_kernel(const T* __restrict__ Hd, int Fh, const float* __restrict__ w2q,
                                                      const float* __restrict__ xlog, int na, int n_cand,
                                                      float* __restrict__ logits, float* __restrict__ probs) {
  pdl_launch_dependents();
  pdl_wait();
  constexpr int VEC = Vec16<T>::N;
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= n_cand) return;
  float acc[16];
#pragma unroll
  for (int k = 0; k < 16; ++k) acc[k] = 0.f;
  const T* h = Hd + static_cast<long long>(row) * Fh;
  for (int f0 = lane * VEC; f0 < Fh; f0 += 32 * VEC) {
    float v[VEC];
    Vec16<T>::load(h + f0, v);
#pragma unroll
    for (int i = 0; i < VEC; ++i) {
      const float* w = w2q + static_cast<long long>(f0 + i) * na;
#pragma unroll
      for (int k = 0; k < 16; ++k)
        if (k < na) acc[k] = fmaf(v[i], __ldg(w + k), acc[k]);
    }
  }
  float lg[16], mx = -INFINITY;
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    if (k < na) {
      float x = acc[k];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
      lg[k] = x + xlog[static_cast<long long>(row) * na + k];
      mx = fmaxf(mx, lg[k]);
    }
  }
  if (lane != 0) return;
  float sum = 0.f;
#pragma unroll
  for (int k = 0; k < 16; ++k)
    if (k < na) {
      logits[static_cast<long long>(row) * na + k] = lg[k];
      sum += __expf(lg[k] - mx);
    }
  if (probs) {
    const float inv = 1.f / sum;
#pragma unroll
    for (int k = 0; k < 16; ++k)
      if (k < na) probs[static_cast<long long>(row) * na + k] = __expf(lg[k] - mx) * inv;
  }
}

}  // namespace

template <int N>
static cudaError_t upload_n(int* dst_a, const int* src_a, int n_a, int* dst_b, const int* src_b, int n_b,
                            cudaStream_t s) {
  UploadArgs<N> a;
  a.dst_a = dst_a;
  a.dst_b = dst_b;
  a.n_a = n_a;
  a.n_b = n_b;
  for (int i = 0; i < n_a; ++i) a.v[i] = src_a[i];
  for (int i = 0; i < n_b; ++i) a.v[n_a + i] = src_b[i];
  const int blocks = (n_a + n_b + 255) / 256;
  prof_begin(KC_MISC, s);
  const cudaError_t err = launch_pdl(upload_kernel<N>, dim3(blocks > 0 ? blocks : 1), dim3(256), 0, s, a);
  prof_end(KC_MISC, s);
  return err;
}

const int kUploadParamInts = 8000;

cudaError_t launch_upload_ints(int* dst_a, const int* src_a, int n_a, int* dst_b, const int* src_b, int n_b,
                               cudaStream_t s) {
  if (n_a < 0 || n_b < 0) return cudaErrorInvalidValue;
  if (n_a + n_b > kUploadParamInts) return cudaErrorNotSupported;
  if (n_a + n_b <= 1000) return upload_n<1000>(dst_a, src_a, n_a, dst_b, src_b, n_b, s);
  return upload_n<8000>(dst_a, src_a, n_a, dst_b, src_b, n_b, s);
}

template <typename T>
cudaError_t launch_dw_gather(const T* Z, const T* cand, T* Z2, int n_cand, int d, int dw_in, cudaStream_t s) {
  if (n_cand == 0) return cudaSuccess;
  prof_begin(KC_HEAD_DW, s);
  cudaError_t e = launch_pdl(dw_gather_kernel<T>, dim3((n_cand + 7) / 8), dim3(256), 0, s, Z, cand, Z2, n_cand, d,
                             dw_in);
  prof_end(KC_HEAD_DW, s);
  return e;
}

template <typename T>
cudaError_t launch_dw_head(const T* Hd, int Fh, const float* w2q, const float* xlog, int na, int n_cand,
                           float* logits, float* probs, cudaStream_t s) {
  if (n_cand == 0) return cudaSuccess;
  if (na > 16) return cudaErrorInvalidValue;
  prof_begin(KC_HEAD_DW, s);
  cudaError_t e = launch_pdl(dw_head_kernel<T>, dim3((n_cand + 7) / 8), dim3(256), 0, s, Hd, Fh, w2q, xlog, na,
                             n_cand, logits, probs);
  prof_end(KC_HEAD_DW, s);
  return e;
}

template <typename T, int CH>
static cudaError_t pack_launch_ch(int na, dim3 grid, cudaStream_t s, const PackArgs& a, const T* cand, const T* ctx,
                                  T* X, int* row_req, int* cand_off_dev, const float* weff_x, const float* cdec,
                                  float* xlog) {
  const int d = a.d;
  if (na <= 1)
    return launch_pdl(pack_kernel<T, 1, CH>, grid, dim3(256), sizeof(float) * 1 * d, s, a, cand, ctx, X, row_req,
                      cand_off_dev, weff_x, cdec, xlog);
  if (na <= 2)
    return launch_pdl(pack_kernel<T, 2, CH>, grid, dim3(256), sizeof(float) * 2 * d, s, a, cand, ctx, X, row_req,
                      cand_off_dev, weff_x, cdec, xlog);
  if (na <= 4)
    return launch_pdl(pack_kernel<T, 4, CH>, grid, dim3(256), sizeof(float) * 4 * d, s, a, cand, ctx, X, row_req,
                      cand_off_dev, weff_x, cdec, xlog);
  if (na <= 8)
    return launch_pdl(pack_kernel<T, 8, CH>, grid, dim3(256), sizeof(float) * 8 * d, s, a, cand, ctx, X, row_req,
                      cand_off_dev, weff_x, cdec, xlog);
  return launch_pdl(pack_kernel<T, 16, CH>, grid, dim3(256), sizeof(float) * 16 * d, s, a, cand, ctx, X, row_req,
                    cand_off_dev, weff_x, cdec, xlog);
}

template <typename T>
cudaError_t launch_pack(int n_req, const int* cand_off_host, int S, int d, int na, const T* cand, const T* ctx, T* X,
                        int* row_req, int* cand_off_dev, const float* weff_x, const float* cdec, float* xlog,
                        cudaStream_t s) {
  if (n_req > kMaxReqParam || na > 16) return cudaErrorInvalidValue;
  PackArgs a;
  a.n_req = n_req;
  a.n_cand = cand_off_host[n_req];
  a.S = S;
  a.d = d;
  a.na = na;
  for (int i = 0; i <= n_req; ++i) a.cand_off[i] = cand_off_host[i];
  const long long n_rows = a.n_cand + static_cast<long long>(n_req) * S;
  if (n_rows == 0) return cudaSuccess;
  const long long rows_per_cta = 8LL * kPackRowsPerWarp;
  const dim3 grid(static_cast<unsigned>((n_rows + rows_per_cta - 1) / rows_per_cta));
  const int ch = (d + 32 * Vec16<T>::N - 1) / (32 * Vec16<T>::N);   // 1, 2 or 4 (d <= 512)
  prof_begin(KC_PACK, s);
  cudaError_t err;
  if (ch == 1) err = pack_launch_ch<T, 1>(na, grid, s, a, cand, ctx, X, row_req, cand_off_dev, weff_x, cdec, xlog);
  else if (ch == 2) err = pack_launch_ch<T, 2>(na, grid, s, a, cand, ctx, X, row_req, cand_off_dev, weff_x, cdec, xlog);
  else err = pack_launch_ch<T, 4>(na, grid, s, a, cand, ctx, X, row_req, cand_off_dev, weff_x, cdec, xlog);
  prof_end(KC_PACK, s);
  return err;
}

cudaError_t launch_rank(int n_req, const int* cand_off_host, const float* probs, int na, int action, int top_k,
                        int* out, cudaStream_t s) {
  if (n_req > kMaxReqParam) return cudaErrorInvalidValue;
  RankArgs a;
  a.n_req = n_req;
  a.na = na;
  a.action = action;
  a.top_k = top_k;
  int max_m = 0;
  for (int i = 0; i <= n_req; ++i) {
    a.cand_off[i] = cand_off_host[i];
    if (i > 0) max_m = max_m > cand_off_host[i] - cand_off_host[i - 1] ? max_m : cand_off_host[i] - cand_off_host[i - 1];
  }
  if (max_m > 32768) return cudaErrorInvalidValue;
  const size_t smem = static_cast<size_t>(max_m > 0 ? max_m : 1) * sizeof(uint32_t);
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(rank_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 32768 * 4);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  // up to 8 CTAs per request (each ranks a slice of its slate against all of
  // it), so that the launch covers the GPU when there are few requests
  int splits = 1;
  while (splits < 8 && static_cast<long long>(splits) * n_req < tc::num_sms() && max_m / (2 * splits) >= 128)
    splits *= 2;
  prof_begin(KC_RANK, s);
  cudaError_t err = launch_pdl(rank_kernel, dim3(n_req, splits), dim3(1024), smem, s, a, probs, out);
  prof_end(KC_RANK, s);
  return err;
}

template cudaError_t launch_dw_gather<float>(const float*, const float*, float*, int, int, int, cudaStream_t);
template cudaError_t launch_dw_gather<__nv_bfloat16>(const __nv_bfloat16*, const __nv_bfloat16*, __nv_bfloat16*, int,
                                                     int, int, cudaStream_t);
template cudaError_t launch_dw_head<float>(const float*, int, const float*, const float*, int, int, float*, float*,
                                           cudaStream_t);
template cudaError_t launch_dw_head<__nv_bfloat16>(const __nv_bfloat16*, int, const float*, const float*, int, int,
                                                   float*, float*, cudaStream_t);
template cudaError_t launch_pack<float>(int, const int*, int, int, int, const float*, const float*, float*, int*,
                                        int*, const float*, const float*, float*, cudaStream_t);
template cudaError_t launch_pack<__nv_bfloat16>(int, const int*, int, int, int, const __nv_bfloat16*,
                                                const __nv_bfloat16*, __nv_bfloat16*, int*, int*, const float*,
                                                const float*, float*, cudaStream_t);

}  // namespace txs
