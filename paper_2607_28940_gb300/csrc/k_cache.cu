// Cache-side kernels: attention pooling of the global anchor, its per-layer
// K/V projection, and the one-time weight preparation of txs_model_create.
//
// Attention pooling (Sec. 4.1.2 local-global set: "attention-pooled global
// representation"; Sec. 5.1 "attention pooling to generate the global token"):
// alpha = softmax_i(phi_i . w_pool / sqrt(d)), g = sum_i alpha_i phi_i.  It is
// kept as an online-softmax state (m = max logit, s = sum exp(logit - m),
// acc = sum exp(logit - m) phi) so that an append (App. D incremental-encoding
// remark) merges new rows without revisiting old ones.  Rows are processed in
// chunks of kPoolChunk (one CTA each); chunk states are merged per request.
#include "txs_internal.cuh"

namespace txs {

constexpr int kPoolChunkV = 128;
extern const int kPoolChunk = kPoolChunkV;

namespace {

template <typename T>
__global__ void __launch_bounds__(256) pool_partial_kernel(const T* __restrict__ phi, const int* __restrict__ seg_off,
                                                           const float* __restrict__ w_pool, int d, float inv_sqrt_d,
                                                           int max_chunks, float* __restrict__ part) {
  __shared__ float z[kPoolChunkV];
  __shared__ float red[8];
  const int r = blockIdx.y, c = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int seg_beg = seg_off[r], seg_end = seg_off[r + 1];
  const int beg = seg_beg + c * kPoolChunkV;
  const int nrows = min(seg_end - beg, kPoolChunkV);
  float* out = part + (static_cast<long long>(r) * max_chunks + c) * (d + 2);
  if (nrows <= 0) {
    for (int i = tid; i < d; i += 256) out[2 + i] = 0.f;
    if (tid == 0) {
      out[0] = -INFINITY;
      out[1] = 0.f;
    }
    return;
  }
  for (int i = warp; i < nrows; i += 8) {
    const T* row = phi + static_cast<long long>(beg + i) * d;
    float dot = 0.f;
    for (int k = lane; k < d; k += 32) dot = fmaf(Elem<T>::load(row + k), __ldg(w_pool + k), dot);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
    if (lane == 0) z[i] = dot * inv_sqrt_d;
  }
  __syncthreads();
  float m = -INFINITY;
  for (int i = tid; i < nrows; i += 256) m = fmaxf(m, z[i]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if (lane == 0) red[warp] = m;
  __syncthreads();
  m = red[0];
#pragma unroll
  for (int w = 1; w < 8; ++w) m = fmaxf(m, red[w]);
  __syncthreads();
  for (int i = tid; i < nrows; i += 256) z[i] = expf(z[i] - m);
  __syncthreads();
  for (int k = tid; k < d; k += 256) {
    float a = 0.f;
    for (int i = 0; i < nrows; ++i) a = fmaf(z[i], Elem<T>::load(phi + static_cast<long long>(beg + i) * d + k), a);
    out[2 + k] = a;
  }
  if (tid == 0) {
    float s = 0.f;
    for (int i = 0; i < nrows; ++i) s += z[i];
    out[0] = m;
    out[1] = s;
  }
}

// Per request: merge the chunk states (and, for an append, the stored state)
// into the stored state and write g = acc / s.
__global__ void __launch_bounds__(256) pool_merge_kernel(const float* __restrict__ part, const int* __restrict__ seg_off,
                                                         int max_chunks, int d, int merge_existing, float* st_m,
                                                         float* st_s, float* st_acc, float* __restrict__ g) {
  const int r = blockIdx.x;
  const int rows = seg_off[r + 1] - seg_off[r];
  const int nch = (rows + kPoolChunkV - 1) / kPoolChunkV;
  const float* p = part + static_cast<long long>(r) * max_chunks * (d + 2);
  const float old_m = merge_existing ? st_m[r] : -INFINITY;
  const float old_s = merge_existing ? st_s[r] : 0.f;
  float M = old_m;
  for (int c = 0; c < nch; ++c) M = fmaxf(M, p[static_cast<long long>(c) * (d + 2)]);
  const float w_old = merge_existing ? expf(old_m - M) : 0.f;
  float S = old_s * w_old;
  for (int c = 0; c < nch; ++c) {
    const float* pc = p + static_cast<long long>(c) * (d + 2);
    S += pc[1] * expf(pc[0] - M);
  }
  for (int k = threadIdx.x; k < d; k += blockDim.x) {
    float a = merge_existing ? st_acc[static_cast<long long>(r) * d + k] * w_old : 0.f;
    for (int c = 0; c < nch; ++c) {
      const float* pc = p + static_cast<long long>(c) * (d + 2);
      a = fmaf(pc[2 + k], expf(pc[0] - M), a);
    }
    st_acc[static_cast<long long>(r) * d + k] = a;
    g[static_cast<long long>(r) * d + k] = a / S;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    st_m[r] = M;
    st_s[r] = S;
  }
}

// Anchor projections for every layer: gkv[blk][r][c] = g[r] . Wt[n] + b[n],
// n = blk * d + c, blk = 2 l + {0: K, 1: V}.  One warp per output column n.
template <typename T>
__global__ void __launch_bounds__(256) global_kv_kernel(const float* __restrict__ g, const T* __restrict__ Wt,
                                                        const float* __restrict__ b, float* __restrict__ gkv, int R,
                                                        int d, int n_total) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = blockIdx.x * 8 + warp;
  if (n >= n_total) return;
  float w[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const int k = lane + 32 * i;
    w[i] = k < d ? Elem<T>::load(Wt + static_cast<long long>(n) * d + k) : 0.f;
  }
  const int blk = n / d, c = n - blk * d;
  const float bias = b[n];
  for (int r = 0; r < R; ++r) {
    const float* gr = g + static_cast<long long>(r) * d;
    float dot = 0.f;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int k = lane + 32 * i;
      if (k < d) dot = fmaf(w[i], gr[k], dot);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
    if (lane == 0) gkv[(static_cast<long long>(blk) * R + r) * d + c] = dot + bias;
  }
}

// Wt[c, r] = W[r, c] for W [rows, cols]; Wt has leading dimension rows.
template <typename T>
__global__ void transpose_kernel(const T* __restrict__ W, T* __restrict__ Wt, int rows, int cols) {
  __shared__ T tile[32][33];
  const int bx = blockIdx.x * 32, by = blockIdx.y * 32;
  for (int j = threadIdx.y; j < 32; j += 8) {
    const int r = by + j, c = bx + threadIdx.x;
    if (r < rows && c < cols) tile[j][threadIdx.x] = W[static_cast<long long>(r) * cols + c];
  }
  __syncthreads();
  for (int j = threadIdx.y; j < 32; j += 8) {
    const int c = bx + j, r = by + threadIdx.x;
    if (r < rows && c < cols) Wt[static_cast<long long>(c) * rows + r] = tile[threadIdx.x][j];
  }
}

template <typename T>
__global__ void to_f32_kernel(const T* __restrict__ src, float* __restrict__ dst, long long n) {
  for (long long i = blockIdx.x * 256LL + threadIdx.x; i < n; i += static_cast<long long>(gridDim.x) * 256)
    dst[i] = Elem<T>::load(src + i);
}

// Head fold (weights only): weff[j, a] = W_dec[j] . Q_dec[a] for j < 2d, and
// cdec[a] = b_dec . Q_dec[a], so logits = [z, x] weff + cdec (Sec. 4.1.3 with a
// linear f_dec).
template <typename T>
__global__ void fold_head_kernel(const T* __restrict__ W_dec, const T* __restrict__ b_dec,
                                 const T* __restrict__ Q_dec, float* __restrict__ weff, float* __restrict__ cdec,
                                 int d, int k) {
  const int t = blockIdx.x * 256 + threadIdx.x;
  if (t >= (2 * d + 1) * k) return;
  const int j = t / k, a = t - j * k;
  const T* w = j < 2 * d ? W_dec + static_cast<long long>(j) * d : b_dec;
  const T* q = Q_dec + static_cast<long long>(a) * d;
  float s = 0.f;
  for (int c = 0; c < d; ++c) s = fmaf(Elem<T>::load(w + c), Elem<T>::load(q + c), s);
  if (j < 2 * d) weff[static_cast<long long>(j) * k + a] = s;
  else cdec[a] = s;
}

// Order-independent 64-bit content hash: sum over 32-bit words of a
// splitmix64-style finaliser of (word, index, salt).
__global__ void hash_kernel(const uint32_t* __restrict__ p, long long n_words, uint64_t salt,
                            unsigned long long* out) {
  uint64_t acc = 0;
  for (long long i = blockIdx.x * 256LL + threadIdx.x; i < n_words; i += static_cast<long long>(gridDim.x) * 256) {
    uint64_t z = (static_cast<uint64_t>(p[i]) << 32 ^ static_cast<uint64_t>(i)) + salt * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    acc += z ^ (z >> 31);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) atomicAdd(out, static_cast<unsigned long long>(acc));
}

}  // namespace

template <typename T>
cudaError_t launch_pool(const T* phi, const int* seg_off, int R, int max_rows, const float* w_pool, int d,
                        int max_chunks, float* part, int merge_existing, float* st_m, float* st_s, float* st_acc,
                        float* g, cudaStream_t s) {
  const int chunks = (max_rows + kPoolChunkV - 1) / kPoolChunkV;
  if (chunks > max_chunks) return cudaErrorInvalidValue;
  prof_begin(KC_POOL, s);
  if (chunks > 0) {
    pool_partial_kernel<T><<<dim3(chunks, R), 256, 0, s>>>(phi, seg_off, w_pool, d, 1.0f / sqrtf(static_cast<float>(d)),
                                                          max_chunks, part);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
  }
  pool_merge_kernel<<<R, 256, 0, s>>>(part, seg_off, max_chunks, d, merge_existing, st_m, st_s, st_acc, g);
  cudaError_t err = cudaGetLastError();
  prof_end(KC_POOL, s);
  return err;
}

template <typename T>
cudaError_t launch_global_kv(const float* g, const T* Wt_kv, const float* b_kv, float* gkv, int R, int d, int n_layers,
                             cudaStream_t s) {
  if (d > 512) return cudaErrorInvalidValue;
  const int n_total = 2 * n_layers * d;
  prof_begin(KC_GLOBAL_KV, s);
  global_kv_kernel<T><<<(n_total + 7) / 8, 256, 0, s>>>(g, Wt_kv, b_kv, gkv, R, d, n_total);
  cudaError_t err = cudaGetLastError();
  prof_end(KC_GLOBAL_KV, s);
  return err;
}

template <typename T>
cudaError_t launch_transpose(const T* W, T* Wt, int rows, int cols, cudaStream_t s) {
  dim3 grid((cols + 31) / 32, (rows + 31) / 32);
  transpose_kernel<T><<<grid, dim3(32, 8), 0, s>>>(W, Wt, rows, cols);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_to_f32(const T* src, float* dst, long long n, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  const long long blocks = (n + 255) / 256;
  to_f32_kernel<T><<<static_cast<int>(blocks < 4096 ? blocks : 4096), 256, 0, s>>>(src, dst, n);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_fold_head(const T* W_dec, const T* b_dec, const T* Q_dec, float* weff, float* cdec, int d, int k,
                             cudaStream_t s) {
  const int n = (2 * d + 1) * k;
  fold_head_kernel<T><<<(n + 255) / 256, 256, 0, s>>>(W_dec, b_dec, Q_dec, weff, cdec, d, k);
  return cudaGetLastError();
}

cudaError_t launch_hash(const void* p, long long bytes, uint64_t salt, unsigned long long* out, cudaStream_t s) {
  const long long words = bytes / 4;
  if (words == 0) return cudaSuccess;
  const long long blocks = (words + 255) / 256;
  hash_kernel<<<static_cast<int>(blocks < 1024 ? blocks : 1024), 256, 0, s>>>(static_cast<const uint32_t*>(p), words,
                                                                              salt, out);
  return cudaGetLastError();
}

#define TXS_INST(T)                                                                                                 \
  template cudaError_t launch_pool<T>(const T*, const int*, int, int, const float*, int, int, float*, int, float*, \
                                      float*, float*, float*, cudaStream_t);                                        \
  template cudaError_t launch_global_kv<T>(const float*, const T*, const float*, float*, int, int, int,            \
                                           cudaStream_t);                                                           \
  template cudaError_t launch_transpose<T>(const T*, T*, int, int, cudaStream_t);                                  \
  template cudaError_t launch_to_f32<T>(const T*, float*, long long, cudaStream_t);                                \
  template cudaError_t launch_fold_head<T>(const T*, const T*, const T*, float*, float*, int, int, cudaStream_t);
TXS_INST(float)
TXS_INST(__nv_bfloat16)
#undef TXS_INST

}  // namespace txs
