// C ABI of libtxs: host-side validation, handle management and the order of
// kernel launches for the cache build, the incremental append, candidate
// scoring and ranking.  Every step of the path runs in the kernels of this
// library; the host only checks arguments, sizes buffers and enqueues work.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <type_traits>
#include <vector>

#include "txs_internal.cuh"

namespace txs {

// ------------------------------------------------------------------ profiler

namespace {
struct ProfRec {
  cudaEvent_t a, b;
  int cls;
};
struct Profiler {
  bool on = false;
  std::vector<ProfRec> recs;
  std::vector<cudaEvent_t> pool;
  int open_cls = -1;
  cudaEvent_t ev() {
    if (!pool.empty()) {
      cudaEvent_t e = pool.back();
      pool.pop_back();
      return e;
    }
    cudaEvent_t e;
    cudaEventCreate(&e);
    return e;
  }
};
Profiler g_prof;
thread_local std::string g_last_error;

void set_error(const char* where, cudaError_t e) {
  g_last_error = std::string(where) + ": " + cudaGetErrorString(e);
}
void set_error(const char* msg) { g_last_error = msg; }
}  // namespace

void prof_begin(int cls, cudaStream_t s) {
  if (!g_prof.on) return;
  ProfRec r{g_prof.ev(), g_prof.ev(), cls};
  cudaEventRecord(r.a, s);
  g_prof.recs.push_back(r);
}

void prof_end(int cls, cudaStream_t s) {
  if (!g_prof.on || g_prof.recs.empty()) return;
  cudaEventRecord(g_prof.recs.back().b, s);
  (void)cls;
}

// ------------------------------------------------------------------ handles

struct LayerW {
  void *Wt_qkv, *Wt_os, *Wt_q, *Wt_oc, *Wt_1, *Wt_2;  // transposed weights [d_out, d_in]
  float *b_qkv, *b_os, *g1, *be1, *b_q, *b_oc, *g2, *be2, *b_1, *b_2, *g3, *be3;
  // the QKV projection with its output columns grouped per head, [q_h | k_h | v_h]
  // (bf16 models with d_h = 64; null otherwise): the fused serving attention
  void* Wt_qkv_h = nullptr;
  float* b_qkv_h = nullptr;
};

}  // namespace txs

struct txs_model {
  txs_config cfg;
  int es = 0;                    // bytes per stored element
  std::vector<void*> allocs;
  std::vector<txs::LayerW> layers;
  void* Wt_kv = nullptr;         // [2 nL dkv, d]: rows (l, K|V, c)
  float* b_kv = nullptr;         // [2 nL dkv]
  float* w_pool = nullptr;       // [d]
  float* weff = nullptr;         // [2d, k]
  float* cdec = nullptr;         // [k]
  void *Wt_c1 = nullptr, *Wt_c2 = nullptr;  // candidate MLP, transposed: [Fc, d], [d, Fc]
  float *b_c1 = nullptr, *b_c2 = nullptr;
  void* Wt_d1 = nullptr;         // Deep & Wide deep FFN layer 1, transposed: [Fh, 2d - dw_in]
  float *b_d1 = nullptr, *w2q = nullptr;  // [Fh], W_d2 Q_deep^T [Fh, k]
  int* status = nullptr;         // device status word
  uint64_t hash = 0;
};

struct txs_kv_cache {
  int n_req = 0, n_layers = 0, d = 0, es = 0, cap_extra = 0;
  int dkv = 0;                           // width of a cached row: n_kv_heads * d_head
  uint64_t model_hash = 0;
  long long cap_total = 0;
  std::vector<int> h_off, h_len, h_cap;  // capacity offsets [R+1], lengths, capacities
  int* h_stage = nullptr;                // pinned staging ring for offset uploads
  int stage_ints = 0;                    // ints per ring slot
  int stage_next = 0;
  cudaEvent_t stage_ev[4] = {nullptr, nullptr, nullptr, nullptr};
  int* d_off = nullptr;                  // [R+1]
  int* d_len = nullptr;                  // [R]
  int* d_in_off = nullptr;               // [R+1] offsets of the rows being projected
  int* d_dst0 = nullptr;                 // [R]   first cache row they go to
  void* kv = nullptr;                    // [nL][2][cap_total][dkv] model dtype
  float *pool_m = nullptr, *pool_s = nullptr, *pool_acc = nullptr, *g = nullptr;
  float* gkv = nullptr;                  // [nL][2][R][dkv] fp32
  float* part = nullptr;                 // pooling chunk states
  int* pool_cnt = nullptr;               // [R] chunk arrivals (zero between calls)
  int max_chunks = 0;
  std::vector<void*> allocs;
};

namespace txs {
namespace {

bool cfg_ok(const txs_config& c, std::string* why) {
  auto bad = [&](const char* m) {
    *why = m;
    return false;
  };
  if (c.dtype != TXS_FP32 && c.dtype != TXS_BF16) return bad("dtype");
  if (c.attn_mode != TXS_ATTN_LOCAL_GLOBAL && c.attn_mode != TXS_ATTN_FULL) return bad("attn_mode");
  if (c.n_layers < 1 || c.n_layers > 64) return bad("n_layers");
  if (c.n_heads < 1 || c.d_model % c.n_heads) return bad("n_heads");
  const int dh = c.d_model / c.n_heads;
  if (dh != 32 && dh != 64) return bad("d_head must be 32 or 64");
  if (c.dtype == TXS_BF16) {
    if (c.d_model != 64 && c.d_model != 128 && c.d_model != 256 && c.d_model != 512) return bad("d_model (bf16)");
  } else if (c.d_model % 32 || c.d_model > 512 || c.d_model < 32) {
    return bad("d_model (fp32)");
  }
  if (c.d_ff < 64 || c.d_ff % 64 || c.d_ff > 16384) return bad("d_ff");
  if (c.n_actions < 1 || c.n_actions > 16) return bad("n_actions");
  if (c.n_ctx < 0 || c.n_ctx > 8) return bad("n_ctx");
  if (c.l_local < 1) return bad("l_local");
  if (!(c.ln_eps > 0.f) || !std::isfinite(c.ln_eps)) return bad("ln_eps");
  if (c.n_kv_heads < 0 || (c.n_kv_heads > 0 && c.n_heads % c.n_kv_heads)) return bad("n_kv_heads");
  if (c.cand_mlp_hidden < 0 || c.cand_mlp_hidden % 64 || c.cand_mlp_hidden > 16384) return bad("cand_mlp_hidden");
  if (c.head_dw_hidden < 0 || c.head_dw_hidden % 64 || c.head_dw_hidden > 16384) return bad("head_dw_hidden");
  if (c.head_dw_hidden > 0) {
    if (c.head_dw_in < 0 || c.head_dw_in > c.d_model || c.head_dw_in % 64) return bad("head_dw_in");
    if (c.head_dw_out < 0 || c.head_dw_out >= c.d_model) return bad("head_dw_out");
  }
  return true;
}

// Width of a cached K or V row: n_kv_heads * d_head (d_model for n_kv_heads 0).
int kv_dim(const txs_config& c) { return (c.n_kv_heads ? c.n_kv_heads : c.n_heads) * (c.d_model / c.n_heads); }

// offsets[0] == 0, non-decreasing (strictly if `strict`), last <= INT32_MAX
bool offsets_ok(const int32_t* off, int n, bool strict) {
  if (!off || n < 0 || off[0] != 0) return false;
  for (int i = 0; i < n; ++i) {
    if (off[i + 1] < off[i]) return false;
    if (strict && off[i + 1] == off[i]) return false;
  }
  return true;
}

template <typename T>
T* dalloc(std::vector<void*>& list, size_t bytes, cudaError_t* err) {
  void* p = nullptr;
  if (bytes == 0) bytes = 16;
  *err = cudaMalloc(&p, bytes);
  if (*err != cudaSuccess) return nullptr;
  list.push_back(p);
  return static_cast<T*>(p);
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

struct ScoreLayout {
  size_t row_req, cand_off, X, QKV, A, X1, X2, Hf, xlog, tmp, total;
};

ScoreLayout score_layout(const txs_config& c, int es, int n_req, long long n_cand) {
  const long long N = n_cand + static_cast<long long>(n_req) * c.n_ctx;
  const size_t d = c.d_model, F = c.d_ff;
  ScoreLayout L{};
  size_t o = 0;
  auto take = [&](size_t bytes) {
    size_t at = o;
    o = align256(o + bytes);
    return at;
  };
  L.row_req = take(N * 4);
  L.cand_off = take((n_req + 1) * 4);
  L.X = take(N * d * es);
  L.QKV = take(N * 3 * d * es);
  L.A = take(N * d * es);
  L.X1 = take(N * d * es);
  L.X2 = take(N * d * es);
  L.Hf = take(N * std::max({F, static_cast<size_t>(c.cand_mlp_hidden), static_cast<size_t>(c.head_dw_hidden)}) * es);
  L.xlog = take(n_cand * c.n_actions * 4);
  L.tmp = take(c.dtype == TXS_FP32 ? N * d * 4 : 0);
  L.total = o;
  return L;
}

// One dense projection C = A W (+ epilogue) in the model's dtype: bf16 on the
// tensor cores, fp32 on the CUDA cores.
cudaError_t gemm(const txs_model* m, const void* A, long long lda, const void* Bt, EpiArgs e, float* tmp,
                 cudaStream_t s, int cls) {
  e.status = m->status;
  if (m->cfg.dtype == TXS_BF16)
    return launch_gemm_tc(static_cast<const __nv_bfloat16*>(A), lda, static_cast<const __nv_bfloat16*>(Bt), e, s, cls);
  return launch_gemm_simt<float>(static_cast<const float*>(A), lda, static_cast<const float*>(Bt), e, tmp, s, cls);
}

EpiArgs epi_base(int epi, long long M, int N, int K) {
  EpiArgs e;
  std::memset(&e, 0, sizeof(e));
  e.epi = epi;
  e.M = static_cast<int>(M);
  e.N = N;
  e.K = K;
  return e;
}

txs_status fail_cuda(const char* where, cudaError_t e) {
  set_error(where, e);
  return TXS_ERR_CUDA;
}

#define TXS_CK(call)                                      \
  do {                                                    \
    cudaError_t e_ = (call);                              \
    if (e_ != cudaSuccess) return fail_cuda(#call, e_);   \
  } while (0)

template <typename T>
txs_status model_prepare(txs_model* m, const void* const* w, cudaStream_t s) {
  const txs_config& c = m->cfg;
  const int d = c.d_model, F = c.d_ff, nL = c.n_layers, k = c.n_actions, dkv = kv_dim(c);
  cudaError_t err;
  auto wt = [&](int rows, int cols) { return dalloc<T>(m->allocs, size_t(rows) * cols * sizeof(T), &err); };
  auto vf = [&](int n) { return dalloc<float>(m->allocs, size_t(n) * 4, &err); };
  auto W = [&](int l, int i) { return static_cast<const T*>(w[l * TXS_WEIGHTS_PER_LAYER + i]); };
  m->Wt_kv = wt(2 * nL * dkv, d);
  if (!m->Wt_kv) return fail_cuda("cudaMalloc", err);
  m->b_kv = vf(2 * nL * dkv);
  if (!m->b_kv) return fail_cuda("cudaMalloc", err);
  for (int l = 0; l < nL; ++l) {
    LayerW L;
    T* p;
    // transposed weights (K-major B operands)
    if (!(p = wt(3 * d, d))) return fail_cuda("cudaMalloc", err);
    TXS_CK(launch_transpose<T>(W(l, 0), p, d, 3 * d, s));
    L.Wt_qkv = p;
    if (!(p = wt(d, d))) return fail_cuda("cudaMalloc", err);
    TXS_CK(launch_transpose<T>(W(l, 2), p, d, d, s));
    L.Wt_os = p;
    if (!(p = wt(d, d))) return fail_cuda("cudaMalloc", err);
    TXS_CK(launch_transpose<T>(W(l, 6), p, d, d, s));
    L.Wt_q = p;
    if (!(p = wt(d, d))) return fail_cuda("cudaMalloc", err);
    TXS_CK(launch_transpose<T>(W(l, 12), p, d, d, s));
    L.Wt_oc = p;
    if (!(p = wt(F, d))) return fail_cuda("cudaMalloc", err);
    TXS_CK(launch_transpose<T>(W(l, 16), p, d, F, s));
    L.Wt_1 = p;
    if (!(p = wt(d, F))) return fail_cuda("cudaMalloc", err);
    TXS_CK(launch_transpose<T>(W(l, 18), p, F, d, s));
    L.Wt_2 = p;
    T* kv = static_cast<T*>(m->Wt_kv);
    TXS_CK(launch_transpose<T>(W(l, 8), kv + size_t(2 * l) * dkv * d, d, dkv, s));
    TXS_CK(launch_transpose<T>(W(l, 10), kv + size_t(2 * l + 1) * dkv * d, d, dkv, s));
    // vectors in fp32
    float** dst[] = {&L.b_qkv, &L.b_os, &L.g1, &L.be1, &L.b_q, &L.b_oc, &L.g2, &L.be2,
                     &L.b_1, &L.b_2, &L.g3, &L.be3};
    const int idx[] = {1, 3, 4, 5, 7, 13, 14, 15, 17, 19, 20, 21};
    const int len[] = {3 * d, d, d, d, d, d, d, d, F, d, d, d};
    for (int i = 0; i < 12; ++i) {
      float* v = vf(len[i]);
      if (!v) return fail_cuda("cudaMalloc", err);
      TXS_CK(launch_to_f32<T>(W(l, idx[i]), v, len[i], s));
      *dst[i] = v;
    }
    TXS_CK(launch_to_f32<T>(W(l, 9), m->b_kv + size_t(2 * l) * dkv, dkv, s));
    TXS_CK(launch_to_f32<T>(W(l, 11), m->b_kv + size_t(2 * l + 1) * dkv, dkv, s));
    if (std::is_same<T, __nv_bfloat16>::value && d / c.n_heads == 64 && 3 * d <= 1536) {
      // rows (h, j, i) of the per-head copy = rows (j d + h 64 + i) of Wt_qkv
      const int H = c.n_heads, dh = 64;
      T* ph = wt(3 * d, d);
      float* bh = vf(3 * d);
      if (!ph || !bh) return fail_cuda("cudaMalloc", err);
      for (int h = 0; h < H; ++h)
        for (int j = 0; j < 3; ++j) {
          TXS_CK(cudaMemcpyAsync(ph + size_t(h * 3 * dh + j * dh) * d, static_cast<T*>(L.Wt_qkv) + size_t(j * d + h * dh) * d,
                                 size_t(dh) * d * sizeof(T), cudaMemcpyDeviceToDevice, s));
          TXS_CK(cudaMemcpyAsync(bh + h * 3 * dh + j * dh, L.b_qkv + j * d + h * dh, dh * sizeof(float),
                                 cudaMemcpyDeviceToDevice, s));
        }
      L.Wt_qkv_h = ph;
      L.b_qkv_h = bh;
    }
    m->layers.push_back(L);
  }
  const void* const* head = w + nL * TXS_WEIGHTS_PER_LAYER;
  if (!(m->w_pool = vf(d))) return fail_cuda("cudaMalloc", err);
  TXS_CK(launch_to_f32<T>(static_cast<const T*>(head[0]), m->w_pool, d, s));
  if (!(m->weff = vf(2 * d * k))) return fail_cuda("cudaMalloc", err);
  if (!(m->cdec = vf(k))) return fail_cuda("cudaMalloc", err);
  const int Fc = c.cand_mlp_hidden, Fh = c.head_dw_hidden;
  const void* const* cm = head + TXS_HEAD_WEIGHTS;
  const void* const* dw = cm + (Fc ? 4 : 0);
  if (!Fh) {
    TXS_CK(launch_fold_head<T>(static_cast<const T*>(head[1]), static_cast<const T*>(head[2]),
                               static_cast<const T*>(head[3]), m->weff, m->cdec, d, k, s));
  } else {
    // Deep & Wide f_dec: the wide part and both biases fold into the x-part
    // weights and constant the pack kernel evaluates; W_d2 folds with Q_dec
    const int a = c.head_dw_in;
    TXS_CK(cudaMemsetAsync(m->weff, 0, sizeof(float) * d * k, s));
    if (!(m->w2q = vf(size_t(Fh) * k)) || !(m->b_d1 = vf(Fh)) || !(m->Wt_d1 = wt(Fh, 2 * d - a)))
      return fail_cuda("cudaMalloc", err);
    TXS_CK(launch_fold_dw<T>(static_cast<const T*>(dw[0]), static_cast<const T*>(dw[1]),
                             static_cast<const T*>(dw[4]), static_cast<const T*>(dw[5]),
                             static_cast<const T*>(head[3]), m->weff + size_t(d) * k, m->cdec, m->w2q, d, a,
                             c.head_dw_out, Fh, k, s));
    TXS_CK(launch_transpose<T>(static_cast<const T*>(dw[2]), static_cast<T*>(m->Wt_d1), 2 * d - a, Fh, s));
    TXS_CK(launch_to_f32<T>(static_cast<const T*>(dw[3]), m->b_d1, Fh, s));
  }
  // candidate-to-query MLP (optional)
  if (Fc) {
    if (!(m->Wt_c1 = wt(Fc, d)) || !(m->Wt_c2 = wt(d, Fc)) || !(m->b_c1 = vf(Fc)) || !(m->b_c2 = vf(d)))
      return fail_cuda("cudaMalloc", err);
    TXS_CK(launch_transpose<T>(static_cast<const T*>(cm[0]), static_cast<T*>(m->Wt_c1), d, Fc, s));
    TXS_CK(launch_transpose<T>(static_cast<const T*>(cm[2]), static_cast<T*>(m->Wt_c2), Fc, d, s));
    TXS_CK(launch_to_f32<T>(static_cast<const T*>(cm[1]), m->b_c1, Fc, s));
    TXS_CK(launch_to_f32<T>(static_cast<const T*>(cm[3]), m->b_c2, d, s));
  }
  // content hash of config and every input tensor
  unsigned long long* dh = dalloc<unsigned long long>(m->allocs, 8, &err);
  if (!dh) return fail_cuda("cudaMalloc", err);
  TXS_CK(cudaMemsetAsync(dh, 0, 8, s));
  const size_t es = sizeof(T);
  for (int l = 0; l < nL; ++l) {
    const size_t n[TXS_WEIGHTS_PER_LAYER] = {size_t(d) * 3 * d, 3 * size_t(d), size_t(d) * d, size_t(d), size_t(d),
                                             size_t(d), size_t(d) * d, size_t(d), size_t(d) * dkv, size_t(dkv),
                                             size_t(d) * dkv, size_t(dkv), size_t(d) * d, size_t(d), size_t(d), size_t(d),
                                             size_t(d) * F, size_t(F), size_t(F) * d, size_t(d), size_t(d), size_t(d)};
    for (int i = 0; i < TXS_WEIGHTS_PER_LAYER; ++i)
      TXS_CK(launch_hash(W(l, i), static_cast<long long>(n[i] * es), uint64_t(l) * 64 + i + 1, dh, s));
  }
  const size_t nh[TXS_HEAD_WEIGHTS] = {size_t(d), 2 * size_t(d) * d, size_t(d), size_t(k) * d};
  for (int i = 0; i < TXS_HEAD_WEIGHTS; ++i)
    if (!Fh || (i != 1 && i != 2))  // W_dec, b_dec are unused with the Deep & Wide head
      TXS_CK(launch_hash(head[i], static_cast<long long>(nh[i] * es), 100000 + i, dh, s));
  if (Fc) {
    const size_t nc[4] = {size_t(d) * Fc, size_t(Fc), size_t(Fc) * d, size_t(d)};
    for (int i = 0; i < 4; ++i) TXS_CK(launch_hash(cm[i], static_cast<long long>(nc[i] * es), 200000 + i, dh, s));
  }
  if (Fh) {
    const size_t a = c.head_dw_in, o = c.head_dw_out;
    const size_t nd[6] = {a * o, o, (2 * size_t(d) - a) * Fh, size_t(Fh), size_t(Fh) * (d - o), size_t(d) - o};
    for (int i = 0; i < 6; ++i)
      if (nd[i]) TXS_CK(launch_hash(dw[i], static_cast<long long>(nd[i] * es), 500000 + i, dh, s));
  }
  unsigned long long hv = 0;
  TXS_CK(cudaMemcpyAsync(&hv, dh, 8, cudaMemcpyDeviceToHost, s));
  TXS_CK(cudaStreamSynchronize(s));
  uint64_t h = hv;
  const int32_t cf[] = {c.d_model, c.n_heads, c.d_ff, c.n_layers, c.n_actions, c.n_ctx, c.l_local, c.attn_mode,
                        c.dtype, kv_dim(c), c.cand_mlp_hidden, c.head_dw_hidden, c.head_dw_in, c.head_dw_out};
  for (int32_t v : cf) h = (h ^ static_cast<uint64_t>(static_cast<uint32_t>(v))) * 0x100000001B3ull;
  uint32_t eps_bits;
  std::memcpy(&eps_bits, &c.ln_eps, 4);
  h = (h ^ eps_bits) * 0x100000001B3ull;
  m->hash = h;
  return TXS_OK;
}

// Next slot of the cache's pinned staging ring, once the copy that last used it
// has run (copies from pinned memory are asynchronous, so a slot is reused
// only after its event has completed).
int* stage_slot(txs_kv_cache* c, cudaStream_t s, cudaEvent_t** ev) {
  const int i = c->stage_next;
  c->stage_next = (i + 1) & 3;
  cudaEventSynchronize(c->stage_ev[i]);
  *ev = &c->stage_ev[i];
  return c->h_stage + static_cast<size_t>(i) * c->stage_ints;
}

// Upload n ints from a staging slot to dst on stream s.
cudaError_t stage_upload(txs_kv_cache* c, int* dst, const int* src, int n, cudaStream_t s) {
  cudaEvent_t* ev;
  int* slot = stage_slot(c, s, &ev);
  std::memcpy(slot, src, sizeof(int) * n);
  cudaError_t err = cudaMemcpyAsync(dst, slot, sizeof(int) * n, cudaMemcpyHostToDevice, s);
  if (err != cudaSuccess) return err;
  return cudaEventRecord(*ev, s);
}

// Upload [in_off (R+1) | dst0 (R)] and the lengths after the call (R): by
// kernel parameters when they fit (capturable), else through pinned memory.
cudaError_t upload_call(txs_kv_cache* c, const std::vector<int>& up, const std::vector<int>& len, cudaStream_t s) {
  const int n_req = c->n_req;
  cudaError_t err = launch_upload_ints(c->d_in_off, up.data(), 2 * n_req + 1, c->d_len, len.data(), n_req, s);
  if (err != cudaErrorNotSupported) return err;
  if ((err = stage_upload(c, c->d_in_off, up.data(), 2 * n_req + 1, s)) != cudaSuccess) return err;
  return stage_upload(c, c->d_len, len.data(), n_req, s);
}

template <typename T>
txs_status project_rows(txs_model* m, txs_kv_cache* c, int n_req, const int32_t* in_off, const void* rows,
                        bool append, cudaStream_t s, bool project_anchor = true) {
  const txs_config& cf = m->cfg;
  const int d = cf.d_model, nL = cf.n_layers;
  const long long total = in_off[n_req];
  // [in_off (R+1) | dst0 (R)] and the new lengths in one upload
  std::vector<int> up(2 * n_req + 1), len(n_req);
  int max_rows = 0;
  for (int r = 0; r <= n_req; ++r) up[r] = in_off[r];
  for (int r = 0; r < n_req; ++r) {
    up[n_req + 1 + r] = c->h_off[r] + (append ? c->h_len[r] : 0);
    len[r] = (append ? c->h_len[r] : 0) + in_off[r + 1] - in_off[r];
    max_rows = std::max(max_rows, in_off[r + 1] - in_off[r]);
  }
  // the tensor-core projection carries the offsets by value and publishes
  // them; otherwise a separate upload comes first
  const bool by_value = std::is_same<T, __nv_bfloat16>::value && total > 0 && n_req <= kKvParamReq;
  if (!by_value) TXS_CK(upload_call(c, up, len, s));
  if (total > 0) {
    const int dkv = c->dkv;
    EpiArgs e = epi_base(EPI_KV, total, 2 * nL * dkv, d);
    if (by_value) {
      e.kv_host_up = up.data();
      e.kv_host_len = len.data();
      e.kv_dev_up = c->d_in_off;
      e.kv_dev_len = c->d_len;
    }
    e.bias = m->b_kv;
    e.out = c->kv;
    e.ldo = dkv;
    e.seg_off = c->d_in_off;
    e.dst_row0 = c->d_dst0;
    e.n_seg = n_req;
    e.col_blk = dkv;
    e.col_blk_stride = c->cap_total * dkv;
    TXS_CK(gemm(m, rows, d, m->Wt_kv, e, nullptr, s, KC_GEMM_KV));
  }
  TXS_CK(launch_pool<T>(static_cast<const T*>(rows), c->d_in_off, n_req, max_rows, m->w_pool, d, c->max_chunks,
                        c->part, append ? 1 : 0, c->pool_m, c->pool_s, c->pool_acc, c->g, c->pool_cnt, m->status, s));
  if (project_anchor)
    TXS_CK(launch_anchor_proj<T>(c->g, static_cast<const T*>(m->Wt_kv), m->b_kv, c->gkv, n_req, d, c->dkv, nL, s));
  return TXS_OK;
}

// What one scoring pass reads of the cache: unit r (a request, or an event of
// a user) sees rows [off[r], off[r] + len[r]) of every layer's K/V and the
// anchor projections gkv[l][0|1][r].
struct KvView {
  const void* kv;          // [nL][2][cap_total][dkv]
  long long cap_total;
  const int* off;          // device [n]
  const int* len;          // device [n]
  const float* gkv;        // device [nL][2][n][dkv]
  cudaEvent_t ready = nullptr;  // recorded after the cache's last write (may be null)
};

template <typename T>
txs_status score_impl(txs_model* m, const KvView& c, int n_req, const int32_t* cand_off, const void* cand_tok,
                      const void* ctx_tok, void* ws, float* logits, float* probs, cudaStream_t s) {
  const txs_config& cf = m->cfg;
  const int d = cf.d_model, F = cf.d_ff, H = cf.n_heads, S = cf.n_ctx, k = cf.n_actions;
  const int dkv = kv_dim(cf), Hkv = dkv / (d / H);
  const long long n_cand = cand_off[n_req];
  const long long N = n_cand + static_cast<long long>(n_req) * S;
  const ScoreLayout L = score_layout(cf, sizeof(T), n_req, n_cand);
  uint8_t* base = static_cast<uint8_t*>(ws);
  int* row_req = reinterpret_cast<int*>(base + L.row_req);
  int* cand_off_dev = reinterpret_cast<int*>(base + L.cand_off);
  T* X = reinterpret_cast<T*>(base + L.X);
  T* QKV = reinterpret_cast<T*>(base + L.QKV);
  T* A = reinterpret_cast<T*>(base + L.A);
  T* X1 = reinterpret_cast<T*>(base + L.X1);
  T* X2 = reinterpret_cast<T*>(base + L.X2);
  T* Hf = reinterpret_cast<T*>(base + L.Hf);
  float* xlog = reinterpret_cast<float*>(base + L.xlog);
  float* tmp = reinterpret_cast<float*>(base + L.tmp);

  TXS_CK(launch_pack<T>(n_req, cand_off, S, d, k, static_cast<const T*>(cand_tok), static_cast<const T*>(ctx_tok), X,
                        row_req, cand_off_dev, m->weff + size_t(d) * k, m->cdec, xlog, s));
  // Phi_candidate: the candidate rows of X go through the MLP (the head's
  // x-part above used the raw tokens)
  if (cf.cand_mlp_hidden && n_cand > 0) {
    const int Fc = cf.cand_mlp_hidden;
    EpiArgs e = epi_base(EPI_BIAS_GELU, n_cand, Fc, d);
    e.bias = m->b_c1;
    e.out = Hf;
    e.ldo = Fc;
    TXS_CK(gemm(m, X, d, m->Wt_c1, e, tmp, s, KC_CAND_MLP));
    e = epi_base(EPI_BIAS, n_cand, d, Fc);
    e.bias = m->b_c2;
    e.out = X;
    e.ldo = d;
    TXS_CK(gemm(m, Hf, Fc, m->Wt_c2, e, tmp, s, KC_CAND_MLP));
  }
  const T* kv = static_cast<const T*>(c.kv);
  // LOCAL_GLOBAL attention fused into the query projection (bf16; heads of
  // 32 or 64 columns, 128-column query tiles, windows of at most 15 rows),
  // when there are at least two 128 x 128 tiles per SM to pipeline; smaller
  // batches take the separate query projection and window kernel
  const int dh = d / H;
  const long long q_tiles = (N + 127) / 128 * (d / 128);
  const bool lg_fused = std::is_same<T, __nv_bfloat16>::value && cf.attn_mode == TXS_ATTN_LOCAL_GLOBAL &&
                        (dh == 32 || dh == 64) && d % 128 == 0 && d <= 512 && cf.l_local <= 15 && dkv % 8 == 0 &&
                        q_tiles >= 2LL * tc::num_sms();
  // serving-stream attention fused into the candidate rows' QKV projection
  // (bf16, d_h = 64, at most 8 context rows, when the 256-row x one-head
  // tiles fill the GPU): the context rows are projected and attended first,
  // then each candidate tile's epilogue attends to them and to its own row
  const bool serve_fused = std::is_same<T, __nv_bfloat16>::value && m->layers[0].Wt_qkv_h != nullptr && S <= 8 &&
                           n_cand > 0 && (n_cand + 255) / 256 * H >= tc::num_sms();
  for (int l = 0; l < cf.n_layers; ++l) {
    const LayerW& W = m->layers[l];
    // serving-stream attention (App. B mask), O-projection + residual + LN1
    EpiArgs e;
    if (serve_fused) {
      const long long n_ctx_rows = N - n_cand;   // R S
      if (n_ctx_rows > 0) {
        e = epi_base(EPI_BIAS, n_ctx_rows, 3 * d, d);
        e.bias = W.b_qkv;
        e.out = QKV + n_cand * 3 * d;
        e.ldo = 3 * d;
        TXS_CK(gemm(m, X + n_cand * d, d, W.Wt_qkv, e, tmp, s, KC_GEMM_QKV));
        TXS_CK(launch_serving_attn<T>(QKV + n_cand * 3 * d, A + n_cand * d, row_req + n_cand,
                                      static_cast<int>(n_ctx_rows), 0, S, H, d, s));
      }
      e = epi_base(EPI_SERVE, n_cand, 3 * d, d);
      e.bias = W.b_qkv_h;
      e.out = A;
      e.ldo = d;
      e.srv_ctx = QKV + n_cand * 3 * d;
      e.srv_row_req = row_req;
      e.srv_S = S;
      e.srv_d = d;
      e.srv_scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(d / H));
      TXS_CK(gemm(m, X, d, W.Wt_qkv_h, e, tmp, s, KC_GEMM_QKV));
    } else {
      e = epi_base(EPI_BIAS, N, 3 * d, d);
      e.bias = W.b_qkv;
      e.out = QKV;
      e.ldo = 3 * d;
      TXS_CK(gemm(m, X, d, W.Wt_qkv, e, tmp, s, KC_GEMM_QKV));
      TXS_CK(launch_serving_attn<T>(QKV, A, row_req, static_cast<int>(N), static_cast<int>(n_cand), S, H, d, s));
    }
    e = epi_base(EPI_LN, N, d, d);
    e.bias = W.b_os;
    e.res = X;
    e.ldr = d;
    e.gamma = W.g1;
    e.beta = W.be1;
    e.ln_eps = cf.ln_eps;
    e.out = X1;
    e.ldo = d;
    TXS_CK(gemm(m, A, d, W.Wt_os, e, tmp, s, KC_GEMM_OPROJ));
    // multi-query cross-attention against the shared cache (Sec. 4.1.2)
    const T* Kc = kv + (size_t(2 * l) * c.cap_total) * dkv;
    const T* Vc = kv + (size_t(2 * l + 1) * c.cap_total) * dkv;
    const float* Kg = c.gkv + size_t(2 * l) * n_req * dkv;
    const float* Vg = c.gkv + size_t(2 * l + 1) * n_req * dkv;
    if (lg_fused) {
      // LOCAL_GLOBAL, bf16: the query projection's epilogue attends to each
      // row's window and anchor and writes the attention output (the query
      // never goes to memory).  It reads the cache, so a caller that is still
      // writing the cache on another stream is waited for here.
      if (l == 0 && c.ready) TXS_CK(cudaStreamWaitEvent(s, c.ready, 0));
      e = epi_base(EPI_ATTN_LG, N, d, d);
      e.bias = W.b_q;
      e.out = A;
      e.ldo = d;
      e.att_k = Kc;
      e.att_v = Vc;
      e.att_kg = Kg;
      e.att_vg = Vg;
      e.att_row_req = row_req;
      e.att_kv_off = c.off;
      e.att_kv_len = c.len;
      e.att_dkv = dkv;
      e.att_group = H / Hkv;
      e.att_dh = d / H;
      e.att_l_local = cf.l_local;
      e.att_scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(d / H));
      e.att_n_cand = static_cast<int>(n_cand);
      e.att_q_ctx = QKV;   // free here: the serving attention has read it
      TXS_CK(gemm(m, X1, d, W.Wt_q, e, tmp, s, KC_GEMM_Q_ATTN));
      // the context-token rows (S per request, rows n_cand + r S + j): q from
      // QKV, attention output over their rows of A
      if (S > 0) {
        const cudaError_t err = launch_ctx_attn_lg(
            reinterpret_cast<const __nv_bfloat16*>(QKV), reinterpret_cast<__nv_bfloat16*>(A),
            reinterpret_cast<const __nv_bfloat16*>(Kc), reinterpret_cast<const __nv_bfloat16*>(Vc), n_req,
            static_cast<int>(n_cand), S, c.off, c.len, Kg, Vg, cf.l_local, H, Hkv, d, s);
        if (err != cudaSuccess) return fail_cuda("context-row cross-attention", err);
      }
    } else {
    e = epi_base(EPI_BIAS, N, d, d);
    e.bias = W.b_q;
    e.out = QKV;
    e.ldo = d;
    TXS_CK(gemm(m, X1, d, W.Wt_q, e, tmp, s, KC_GEMM_Q));
    // the first read of the cache: a caller that is still writing it on
    // another stream made everything above overlap with that write
    if (l == 0 && c.ready) TXS_CK(cudaStreamWaitEvent(s, c.ready, 0));
    cudaError_t lg = cudaErrorNotSupported;
    if (cf.attn_mode == TXS_ATTN_LOCAL_GLOBAL)
      lg = launch_cross_attn_lg<T>(QKV, A, Kc, Vc, cand_off_dev, cand_off, n_req, static_cast<int>(n_cand), S,
                                   c.off, c.len, Kg, Vg, cf.l_local, H, Hkv, d, s);
    if (lg != cudaErrorNotSupported) {
      if (lg != cudaSuccess) return fail_cuda("cross-attention", lg);
    } else if constexpr (std::is_same<T, __nv_bfloat16>::value) {
      if (cf.attn_mode == TXS_ATTN_FULL && fa_full_supported(d, H, c.cap_total)) {
        TXS_CK(launch_fa_full(QKV, A, Kc, Vc, c.cap_total, cand_off_dev, cand_off, c.off, c.len, n_req,
                              static_cast<int>(n_cand), S, H, Hkv, d, m->status, s));
      } else {
        TXS_CK(launch_cross_attn<T>(QKV, A, Kc, Vc, row_req, static_cast<int>(N), c.off, c.len, Kg, Vg,
                                    cf.l_local, cf.attn_mode, H, Hkv, d, s));
      }
    } else {
      TXS_CK(launch_cross_attn<T>(QKV, A, Kc, Vc, row_req, static_cast<int>(N), c.off, c.len, Kg, Vg,
                                  cf.l_local, cf.attn_mode, H, Hkv, d, s));
    }
    }
    e = epi_base(EPI_LN, N, d, d);
    e.bias = W.b_oc;
    e.res = X1;
    e.ldr = d;
    e.gamma = W.g2;
    e.beta = W.be2;
    e.ln_eps = cf.ln_eps;
    e.out = X2;
    e.ldo = d;
    TXS_CK(gemm(m, A, d, W.Wt_oc, e, tmp, s, KC_GEMM_OPROJ));
    // FFN with GELU, then residual + LN3 (the last layer also runs the head)
    e = epi_base(EPI_BIAS_GELU, N, F, d);
    e.bias = W.b_1;
    e.out = Hf;
    e.ldo = F;
    TXS_CK(gemm(m, X2, d, W.Wt_1, e, tmp, s, KC_GEMM_FFN1));
    const bool last = l == cf.n_layers - 1 && !cf.head_dw_hidden;  // fused linear head
    e = epi_base(last ? EPI_LN_HEAD : EPI_LN, N, d, F);
    e.bias = W.b_2;
    e.res = X2;
    e.ldr = d;
    e.gamma = W.g3;
    e.beta = W.be3;
    e.ln_eps = cf.ln_eps;
    e.out = X;
    e.ldo = d;
    if (last) {
      e.weff_z = m->weff;
      e.xlog = xlog;
      e.n_act = k;
      e.n_cand_rows = static_cast<int>(n_cand);
      e.logits = logits;
      e.probs = probs;
    }
    TXS_CK(gemm(m, Hf, F, W.Wt_2, e, tmp, s, KC_GEMM_FFN2));
  }
  // Deep & Wide f_dec (App. B): h = GELU([z, x_deep] W_d1 + b_d1) on the
  // candidate rows, logits = x weff_x + cdec (from the pack kernel) + h w2q
  if (cf.head_dw_hidden && n_cand > 0) {
    const int a = cf.head_dw_in, Fh = cf.head_dw_hidden, w2 = 2 * d - a;
    T* Z2 = QKV;  // free after the last layer: [n_cand, 2d - dw_in]
    TXS_CK(launch_dw_gather<T>(X, static_cast<const T*>(cand_tok), Z2, static_cast<int>(n_cand), d, a, s));
    EpiArgs e = epi_base(EPI_BIAS_GELU, n_cand, Fh, w2);
    e.bias = m->b_d1;
    e.out = Hf;
    e.ldo = Fh;
    TXS_CK(gemm(m, Z2, w2, m->Wt_d1, e, tmp, s, KC_HEAD_DW));
    TXS_CK(launch_dw_head<T>(Hf, Fh, m->w2q, xlog, k, static_cast<int>(n_cand), logits, probs, s));
  }
  return TXS_OK;
}

}  // namespace
}  // namespace txs

using namespace txs;

// ------------------------------------------------------------------ C ABI

TXS_API const char* txs_version(void) { return "txs 0.1 (sm_103a)"; }

TXS_API const char* txs_status_string(txs_status s) {
  TXS_TRACE();
  switch (s) {
    case TXS_OK: return "ok";
    case TXS_ERR_INVALID_ARG: return "invalid argument";
    case TXS_ERR_COLD_START: return "cold start: request without behavior rows";
    case TXS_ERR_CAPACITY: return "append exceeds cache capacity";
    case TXS_ERR_STALE_CACHE: return "cache built by another model";
    case TXS_ERR_CUDA: return "CUDA error";
    case TXS_ERR_DEVICE_TIMEOUT: return "device-side wait timed out";
    case TXS_ERR_BOUNDS: return "device-side bounds check failed";
    case TXS_ERR_UNSUPPORTED: return "unsupported shape";
  }
  return "unknown status";
}

TXS_API const char* txs_last_error(void) { return g_last_error.c_str(); }

namespace txs {
void set_last_error(const char* msg) { set_error(msg); }
int model_d(const txs_model* m) { return m->cfg.d_model; }
int model_dtype(const txs_model* m) { return m->cfg.dtype; }
const float* model_w_pool(const txs_model* m) { return m->w_pool; }
}  // namespace txs

TXS_API txs_status txs_model_create(const txs_config* cfg, const void* const* weights, txs_model** out) {
  TXS_TRACE();
  if (!cfg || !weights || !out) return TXS_ERR_INVALID_ARG;
  *out = nullptr;
  std::string why;
  if (!cfg_ok(*cfg, &why)) {
    set_error(why.c_str());
    return TXS_ERR_UNSUPPORTED;
  }
  const int n_dec = cfg->n_layers * TXS_WEIGHTS_PER_LAYER, n_cm = cfg->cand_mlp_hidden ? 4 : 0;
  const int n_w = n_dec + TXS_HEAD_WEIGHTS + n_cm + (cfg->head_dw_hidden ? 6 : 0);
  for (int i = 0; i < n_w; ++i) {
    if (weights[i]) continue;
    const int h = i - n_dec, dwi = i - n_dec - TXS_HEAD_WEIGHTS - n_cm;
    const bool optional = cfg->head_dw_hidden &&
                          (h == 1 || h == 2 ||  // W_dec, b_dec unused with the Deep & Wide head
                           (dwi == 0 && (cfg->head_dw_in == 0 || cfg->head_dw_out == 0)) ||
                           (dwi == 1 && cfg->head_dw_out == 0));
    if (!optional) return TXS_ERR_INVALID_ARG;
  }
  // the weight tensors may still be in flight on any stream of the caller
  cudaError_t pre = cudaDeviceSynchronize();
  if (pre != cudaSuccess) return fail_cuda("cudaDeviceSynchronize", pre);
  txs_model* m = new txs_model();
  m->cfg = *cfg;
  m->es = cfg->dtype == TXS_BF16 ? 2 : 4;
  cudaError_t err;
  m->status = dalloc<int>(m->allocs, 4, &err);
  txs_status st = TXS_OK;
  if (!m->status) st = fail_cuda("cudaMalloc", err);
  if (st == TXS_OK && cudaMemset(m->status, 0, 4) != cudaSuccess) st = TXS_ERR_CUDA;
  cudaStream_t s = nullptr;
  if (st == TXS_OK && cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking) != cudaSuccess) st = TXS_ERR_CUDA;
  if (st == TXS_OK)
    st = cfg->dtype == TXS_BF16 ? model_prepare<__nv_bfloat16>(m, weights, s) : model_prepare<float>(m, weights, s);
  if (s) {
    if (cudaStreamSynchronize(s) != cudaSuccess && st == TXS_OK) st = TXS_ERR_CUDA;
    cudaStreamDestroy(s);
  }
  if (st != TXS_OK) {
    txs_model_destroy(m);
    return st;
  }
  *out = m;
  return TXS_OK;
}

TXS_API void txs_model_destroy(txs_model* m) {
  TXS_TRACE();
  if (!m) return;
  for (void* p : m->allocs) cudaFree(p);
  delete m;
}

TXS_API uint64_t txs_model_hash(const txs_model* m) { return m ? m->hash : 0; }

// A cache of n_req requests of the given lengths (each with capacity_extra
// spare rows), its device arrays allocated and its offsets and lengths
// uploaded; the K/V rows and pooling state are left for the caller to fill.
txs_status make_cache(txs_model* m, int n_req, const int* lengths, int capacity_extra, cudaStream_t s,
                      txs_kv_cache** out) {
  const txs_config& cf = m->cfg;
  const int d = cf.d_model, nL = cf.n_layers;
  txs_kv_cache* c = new txs_kv_cache();
  c->n_req = n_req;
  c->n_layers = nL;
  c->d = d;
  c->dkv = kv_dim(cf);
  c->es = m->es;
  c->cap_extra = capacity_extra;
  c->model_hash = m->hash;
  c->h_off.assign(n_req + 1, 0);
  c->h_len.assign(n_req, 0);
  c->h_cap.assign(n_req, 0);
  long long tot = 0;
  int max_cap = 0;
  for (int r = 0; r < n_req; ++r) {
    c->h_len[r] = lengths[r];
    c->h_cap[r] = c->h_len[r] + capacity_extra;
    max_cap = std::max(max_cap, c->h_cap[r]);
    c->h_off[r] = static_cast<int>(tot);
    tot += c->h_cap[r];
    if (tot > 0x7FFFFFFFLL) {
      delete c;
      return TXS_ERR_UNSUPPORTED;
    }
  }
  c->h_off[n_req] = static_cast<int>(tot);
  c->cap_total = tot;
  c->max_chunks = (max_cap + kPoolChunk - 1) / kPoolChunk;
  cudaError_t err = cudaSuccess;
  txs_status st = TXS_OK;
  auto A = [&](size_t bytes) -> void* {
    if (st != TXS_OK) return nullptr;
    void* p = dalloc<void>(c->allocs, bytes, &err);
    if (!p) st = fail_cuda("cudaMalloc", err);
    return p;
  };
  c->kv = A(size_t(nL) * 2 * tot * c->dkv * m->es);
  // zeroed: a FULL-mode key tile may read rows past a request's length
  // (masked, P = 0), which must hold finite values
  if (st == TXS_OK && (err = cudaMemsetAsync(c->kv, 0, size_t(nL) * 2 * tot * c->dkv * m->es, s)) != cudaSuccess)
    st = fail_cuda("cudaMemsetAsync", err);
  c->d_off = static_cast<int*>(A(4 * (n_req + 1)));
  c->d_len = static_cast<int*>(A(4 * n_req));
  c->d_in_off = static_cast<int*>(A(4 * (2 * n_req + 1)));
  if (st == TXS_OK) c->d_dst0 = c->d_in_off + n_req + 1;
  c->pool_m = static_cast<float*>(A(4 * n_req));
  c->pool_s = static_cast<float*>(A(4 * n_req));
  c->pool_acc = static_cast<float*>(A(size_t(4) * n_req * d));
  c->g = static_cast<float*>(A(size_t(4) * n_req * d));
  c->gkv = static_cast<float*>(A(size_t(4) * nL * 2 * n_req * c->dkv));
  c->part = static_cast<float*>(A(size_t(4) * n_req * c->max_chunks * (d + 2)));
  c->pool_cnt = static_cast<int*>(A(size_t(4) * n_req));
  if (st == TXS_OK && (err = cudaMemsetAsync(c->pool_cnt, 0, size_t(4) * n_req, s)) != cudaSuccess)
    st = fail_cuda("cudaMemsetAsync", err);
  if (st == TXS_OK) {
    c->stage_ints = 2 * n_req + 1;
    if ((err = cudaMallocHost(&c->h_stage, sizeof(int) * 4 * c->stage_ints)) != cudaSuccess) {
      c->h_stage = nullptr;
      st = fail_cuda("cudaMallocHost", err);
    }
    for (int i = 0; i < 4 && st == TXS_OK; ++i)
      if ((err = cudaEventCreateWithFlags(&c->stage_ev[i], cudaEventDisableTiming)) != cudaSuccess)
        st = fail_cuda("cudaEventCreate", err);
  }
  if (st == TXS_OK) {
    if ((err = stage_upload(c, c->d_off, c->h_off.data(), n_req + 1, s)) != cudaSuccess ||
        (err = stage_upload(c, c->d_len, c->h_len.data(), n_req, s)) != cudaSuccess)
      st = fail_cuda("upload", err);
  }
  if (st != TXS_OK) {
    cudaStreamSynchronize(s);
    txs_cache_destroy(c);
    return st;
  }
  *out = c;
  return TXS_OK;
}

TXS_API txs_status txs_build_kv_cache(txs_model* m, int32_t n_req, const int32_t* beh_offsets, const void* beh_enc,
                                      int32_t capacity_extra, void* stream, txs_kv_cache** out) {
  TXS_TRACE();
  if (!m || !out || n_req < 1 || capacity_extra < 0 || !beh_offsets) return TXS_ERR_INVALID_ARG;
  *out = nullptr;
  if (!offsets_ok(beh_offsets, n_req, false)) return TXS_ERR_INVALID_ARG;
  for (int r = 0; r < n_req; ++r)
    if (beh_offsets[r + 1] == beh_offsets[r]) return TXS_ERR_COLD_START;
  if (!beh_enc) return TXS_ERR_INVALID_ARG;
  if (n_req > kMaxReqParam) return TXS_ERR_UNSUPPORTED;
  const txs_config& cf = m->cfg;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  std::vector<int> lengths(n_req);
  for (int r = 0; r < n_req; ++r) lengths[r] = beh_offsets[r + 1] - beh_offsets[r];
  txs_kv_cache* c = nullptr;
  txs_status st = make_cache(m, n_req, lengths.data(), capacity_extra, s, &c);
  if (st != TXS_OK) return st;
  if (st == TXS_OK)
    st = cf.dtype == TXS_BF16 ? project_rows<__nv_bfloat16>(m, c, n_req, beh_offsets, beh_enc, false, s)
                              : project_rows<float>(m, c, n_req, beh_offsets, beh_enc, false, s);
  if (st != TXS_OK) {
    cudaStreamSynchronize(s);
    txs_cache_destroy(c);
    return st;
  }
  *out = c;
  return TXS_OK;
}

// ------------------------------------------------------------------ cache export / import

// Serialised cache (host memory): header, lengths, each layer's K and V rows
// of every request (no spare capacity), then the pooling state (m, s, acc),
// the pooled anchor g and its projections.  Entries are versioned by the
// model hash and a caller-given feature-schema version (App. D cache
// management: versioning and consistency).
namespace {
constexpr char kCacheMagic[8] = {'T', 'X', 'S', 'C', 'A', 'C', 'H', 'E'};
constexpr uint32_t kCacheFormat = 1;
struct CacheHeader {
  char magic[8];
  uint32_t format, schema;
  uint64_t model_hash;
  int32_t n_req, n_layers, d_model, d_kv, elem_bytes, reserved;
  int64_t total_rows;
};
size_t cache_blob_bytes(int n_req, int nL, int d, int dkv, int es, long long rows) {
  return sizeof(CacheHeader) + sizeof(int32_t) * n_req + size_t(nL) * 2 * rows * dkv * es +
         sizeof(float) * (2 * size_t(n_req) + size_t(2) * n_req * d + size_t(nL) * 2 * n_req * dkv);
}
}  // namespace

TXS_API txs_status txs_cache_export_size(const txs_kv_cache* c, size_t* bytes) {
  TXS_TRACE();
  if (!c || !bytes) return TXS_ERR_INVALID_ARG;
  long long rows = 0;
  for (int r = 0; r < c->n_req; ++r) rows += c->h_len[r];
  *bytes = cache_blob_bytes(c->n_req, c->n_layers, c->d, c->dkv, c->es, rows);
  return TXS_OK;
}

TXS_API txs_status txs_cache_export(const txs_kv_cache* c, uint32_t schema_version, void* host_buf, size_t bytes,
                                    void* stream) {
  TXS_TRACE();
  if (!c || !host_buf) return TXS_ERR_INVALID_ARG;
  size_t need = 0;
  txs_cache_export_size(c, &need);
  if (bytes < need) return TXS_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int R = c->n_req, nL = c->n_layers, d = c->d, dkv = c->dkv, es = c->es;
  uint8_t* p = static_cast<uint8_t*>(host_buf);
  CacheHeader h;
  std::memcpy(h.magic, kCacheMagic, 8);
  h.format = kCacheFormat;
  h.schema = schema_version;
  h.model_hash = c->model_hash;
  h.n_req = R;
  h.n_layers = nL;
  h.d_model = d;
  h.d_kv = dkv;
  h.elem_bytes = es;
  h.reserved = 0;
  h.total_rows = 0;
  for (int r = 0; r < R; ++r) h.total_rows += c->h_len[r];
  std::memcpy(p, &h, sizeof(h));
  p += sizeof(h);
  std::memcpy(p, c->h_len.data(), sizeof(int32_t) * R);
  p += sizeof(int32_t) * R;
  cudaError_t err = cudaSuccess;
  const uint8_t* kv = static_cast<const uint8_t*>(c->kv);
  for (int l = 0; l < nL && err == cudaSuccess; ++l)
    for (int w = 0; w < 2 && err == cudaSuccess; ++w)
      for (int r = 0; r < R && err == cudaSuccess; ++r) {
        const size_t n = size_t(c->h_len[r]) * dkv * es;
        const size_t src = ((size_t(2 * l + w) * c->cap_total) + c->h_off[r]) * dkv * es;
        err = cudaMemcpyAsync(p, kv + src, n, cudaMemcpyDeviceToHost, s);
        p += n;
      }
  auto grab = [&](const float* src, size_t n) {
    if (err == cudaSuccess) err = cudaMemcpyAsync(p, src, sizeof(float) * n, cudaMemcpyDeviceToHost, s);
    p += sizeof(float) * n;
  };
  grab(c->pool_m, R);
  grab(c->pool_s, R);
  grab(c->pool_acc, size_t(R) * d);
  grab(c->g, size_t(R) * d);
  grab(c->gkv, size_t(nL) * 2 * R * dkv);
  if (err == cudaSuccess) err = cudaStreamSynchronize(s);
  if (err != cudaSuccess) return fail_cuda("cache export", err);
  return TXS_OK;
}

TXS_API txs_status txs_cache_import(txs_model* m, uint32_t schema_version, const void* host_buf, size_t bytes,
                                    int32_t capacity_extra, void* stream, txs_kv_cache** out) {
  TXS_TRACE();
  if (!m || !host_buf || !out || capacity_extra < 0) return TXS_ERR_INVALID_ARG;
  *out = nullptr;
  if (bytes < sizeof(CacheHeader)) return TXS_ERR_INVALID_ARG;
  CacheHeader h;
  std::memcpy(&h, host_buf, sizeof(h));
  if (std::memcmp(h.magic, kCacheMagic, 8) != 0 || h.format != kCacheFormat) return TXS_ERR_INVALID_ARG;
  // entries of another model or feature schema are stale, never reinterpreted
  if (h.model_hash != m->hash || h.schema != schema_version) return TXS_ERR_STALE_CACHE;
  const txs_config& cf = m->cfg;
  if (h.n_layers != cf.n_layers || h.d_model != cf.d_model || h.d_kv != kv_dim(cf) || h.elem_bytes != m->es)
    return TXS_ERR_STALE_CACHE;
  if (h.n_req < 1 || h.n_req > kMaxReqParam || h.total_rows < 0) return TXS_ERR_INVALID_ARG;
  const int R = h.n_req, nL = h.n_layers, d = h.d_model, dkv = h.d_kv, es = h.elem_bytes;
  if (bytes < sizeof(h) + sizeof(int32_t) * R) return TXS_ERR_INVALID_ARG;
  std::vector<int> len(R);
  std::memcpy(len.data(), static_cast<const uint8_t*>(host_buf) + sizeof(h), sizeof(int32_t) * R);
  long long rows = 0;
  for (int r = 0; r < R; ++r) {
    if (len[r] < 1) return TXS_ERR_INVALID_ARG;
    rows += len[r];
  }
  if (rows != h.total_rows || bytes < cache_blob_bytes(R, nL, d, dkv, es, rows)) return TXS_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  txs_kv_cache* c = nullptr;
  txs_status st = make_cache(m, R, len.data(), capacity_extra, s, &c);
  if (st != TXS_OK) return st;
  const uint8_t* p = static_cast<const uint8_t*>(host_buf) + sizeof(h) + sizeof(int32_t) * R;
  cudaError_t err = cudaSuccess;
  uint8_t* kv = static_cast<uint8_t*>(c->kv);
  for (int l = 0; l < nL && err == cudaSuccess; ++l)
    for (int w = 0; w < 2 && err == cudaSuccess; ++w)
      for (int r = 0; r < R && err == cudaSuccess; ++r) {
        const size_t n = size_t(len[r]) * dkv * es;
        const size_t dst = ((size_t(2 * l + w) * c->cap_total) + c->h_off[r]) * dkv * es;
        err = cudaMemcpyAsync(kv + dst, p, n, cudaMemcpyHostToDevice, s);
        p += n;
      }
  auto put = [&](float* dst, size_t n) {
    if (err == cudaSuccess) err = cudaMemcpyAsync(dst, p, sizeof(float) * n, cudaMemcpyHostToDevice, s);
    p += sizeof(float) * n;
  };
  put(c->pool_m, R);
  put(c->pool_s, R);
  put(c->pool_acc, size_t(R) * d);
  put(c->g, size_t(R) * d);
  put(c->gkv, size_t(nL) * 2 * R * dkv);
  // the host buffer may be released as soon as this returns
  if (err == cudaSuccess) err = cudaStreamSynchronize(s);
  if (err != cudaSuccess) {
    txs_cache_destroy(c);
    return fail_cuda("cache import", err);
  }
  *out = c;
  return TXS_OK;
}

TXS_API void txs_cache_destroy(txs_kv_cache* c) {
  TXS_TRACE();
  if (!c) return;
  for (cudaEvent_t e : c->stage_ev)
    if (e) cudaEventSynchronize(e);
  for (void* p : c->allocs) cudaFree(p);
  for (cudaEvent_t e : c->stage_ev)
    if (e) cudaEventDestroy(e);
  if (c->h_stage) cudaFreeHost(c->h_stage);
  delete c;
}

TXS_API txs_status txs_rebuild_kv_cache(txs_model* m, txs_kv_cache* c, int32_t n_req, const int32_t* beh_offsets,
                                        const void* beh_enc, void* stream) {
  TXS_TRACE();
  if (!m || !c || !beh_offsets) return TXS_ERR_INVALID_ARG;
  if (c->model_hash != m->hash) return TXS_ERR_STALE_CACHE;
  if (n_req != c->n_req || !offsets_ok(beh_offsets, n_req, false)) return TXS_ERR_INVALID_ARG;
  for (int r = 0; r < n_req; ++r) {
    if (beh_offsets[r + 1] == beh_offsets[r]) return TXS_ERR_COLD_START;
    if (beh_offsets[r + 1] - beh_offsets[r] > c->h_cap[r]) return TXS_ERR_CAPACITY;
  }
  if (!beh_enc) return TXS_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  txs_status st = m->cfg.dtype == TXS_BF16 ? project_rows<__nv_bfloat16>(m, c, n_req, beh_offsets, beh_enc, false, s)
                                           : project_rows<float>(m, c, n_req, beh_offsets, beh_enc, false, s);
  if (st != TXS_OK) return st;
  for (int r = 0; r < n_req; ++r) c->h_len[r] = beh_offsets[r + 1] - beh_offsets[r];
  return TXS_OK;
}

TXS_API txs_status txs_rebuild_append_kv_cache(txs_model* m, txs_kv_cache* c, int32_t n_req,
                                               const int32_t* beh_offsets, const void* beh_enc,
                                               const int32_t* new_offsets, const void* new_enc, void* stream) {
  TXS_TRACE();
  if (!m || !c || !beh_offsets || !new_offsets) return TXS_ERR_INVALID_ARG;
  if (c->model_hash != m->hash) return TXS_ERR_STALE_CACHE;
  if (n_req != c->n_req || !offsets_ok(beh_offsets, n_req, false) || !offsets_ok(new_offsets, n_req, false))
    return TXS_ERR_INVALID_ARG;
  for (int r = 0; r < n_req; ++r) {
    if (beh_offsets[r + 1] == beh_offsets[r]) return TXS_ERR_COLD_START;
    if (static_cast<long long>(beh_offsets[r + 1] - beh_offsets[r]) + (new_offsets[r + 1] - new_offsets[r]) >
        c->h_cap[r])
      return TXS_ERR_CAPACITY;
  }
  if (!beh_enc || (new_offsets[n_req] > 0 && !new_enc)) return TXS_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const bool bf16 = m->cfg.dtype == TXS_BF16;
  const bool any_new = new_offsets[n_req] > 0;
  // the rebuild's anchor would be replaced at once: project it only after the append
  txs_status st = bf16 ? project_rows<__nv_bfloat16>(m, c, n_req, beh_offsets, beh_enc, false, s, !any_new)
                       : project_rows<float>(m, c, n_req, beh_offsets, beh_enc, false, s, !any_new);
  if (st != TXS_OK) return st;
  for (int r = 0; r < n_req; ++r) c->h_len[r] = beh_offsets[r + 1] - beh_offsets[r];
  if (!any_new) return TXS_OK;
  st = bf16 ? project_rows<__nv_bfloat16>(m, c, n_req, new_offsets, new_enc, true, s)
            : project_rows<float>(m, c, n_req, new_offsets, new_enc, true, s);
  if (st != TXS_OK) return st;
  for (int r = 0; r < n_req; ++r) c->h_len[r] += new_offsets[r + 1] - new_offsets[r];
  return TXS_OK;
}

TXS_API txs_status txs_append_behavior(txs_model* m, txs_kv_cache* c, int32_t n_req, const int32_t* new_offsets,
                                       const void* new_enc, void* stream) {
  TXS_TRACE();
  if (!m || !c || !new_offsets) return TXS_ERR_INVALID_ARG;
  if (c->model_hash != m->hash) return TXS_ERR_STALE_CACHE;
  if (n_req != c->n_req || !offsets_ok(new_offsets, n_req, false)) return TXS_ERR_INVALID_ARG;
  for (int r = 0; r < n_req; ++r)
    if (static_cast<long long>(c->h_len[r]) + (new_offsets[r + 1] - new_offsets[r]) > c->h_cap[r])
      return TXS_ERR_CAPACITY;
  if (new_offsets[n_req] == 0) return TXS_OK;
  if (!new_enc) return TXS_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  txs_status st = m->cfg.dtype == TXS_BF16 ? project_rows<__nv_bfloat16>(m, c, n_req, new_offsets, new_enc, true, s)
                                           : project_rows<float>(m, c, n_req, new_offsets, new_enc, true, s);
  if (st != TXS_OK) return st;
  for (int r = 0; r < n_req; ++r) c->h_len[r] += new_offsets[r + 1] - new_offsets[r];
  return TXS_OK;
}

TXS_API txs_status txs_cache_lengths(const txs_kv_cache* c, int32_t* out_len) {
  TXS_TRACE();
  if (!c || !out_len) return TXS_ERR_INVALID_ARG;
  for (int r = 0; r < c->n_req; ++r) out_len[r] = c->h_len[r];
  return TXS_OK;
}

TXS_API int32_t txs_cache_n_req(const txs_kv_cache* c) { return c ? c->n_req : 0; }

TXS_API txs_status txs_cache_read_rows(const txs_kv_cache* c, int32_t layer, int32_t which, int32_t req, int32_t row0,
                                       int32_t n_rows, void* dst, void* stream) {
  TXS_TRACE();
  if (!c || !dst || layer < 0 || layer >= c->n_layers || which < 0 || which > 1 || req < 0 || req >= c->n_req ||
      row0 < 0 || n_rows < 0 || static_cast<long long>(row0) + n_rows > c->h_len[req])
    return TXS_ERR_INVALID_ARG;
  if (n_rows == 0) return TXS_OK;
  const size_t row_bytes = size_t(c->dkv) * c->es;
  const size_t blk = size_t(2 * layer + which) * c->cap_total;
  const uint8_t* src = static_cast<const uint8_t*>(c->kv) + (blk + c->h_off[req] + row0) * row_bytes;
  cudaError_t err = cudaMemcpyAsync(dst, src, n_rows * row_bytes, cudaMemcpyDeviceToDevice,
                                    static_cast<cudaStream_t>(stream));
  return err == cudaSuccess ? TXS_OK : fail_cuda("read rows", err);
}

TXS_API txs_status txs_cache_read_anchor(const txs_kv_cache* c, int32_t layer, int32_t which, float* dst,
                                         void* stream) {
  TXS_TRACE();
  if (!c || !dst || which < 0 || which > 2 || (which < 2 && (layer < 0 || layer >= c->n_layers)))
    return TXS_ERR_INVALID_ARG;
  const size_t bytes = size_t(c->n_req) * (which == 2 ? c->d : c->dkv) * 4;
  const float* src = which == 2 ? c->g : c->gkv + size_t(2 * layer + which) * c->n_req * c->dkv;
  cudaError_t err = cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, static_cast<cudaStream_t>(stream));
  return err == cudaSuccess ? TXS_OK : fail_cuda("read anchor", err);
}

TXS_API txs_status txs_score_workspace_size(const txs_model* m, int32_t n_req, int64_t total_cand, size_t* bytes) {
  TXS_TRACE();
  if (!m || !bytes || n_req < 0 || total_cand < 0) return TXS_ERR_INVALID_ARG;
  *bytes = score_layout(m->cfg, m->es, n_req, total_cand).total;
  return TXS_OK;
}

namespace txs {
namespace {
txs_status score_entry(txs_model* m, const txs_kv_cache* c, int32_t n_req, const int32_t* cand_offsets,
                       const void* cand_tok, const void* ctx_tok, void* workspace, size_t workspace_bytes,
                       float* out_logits, float* out_probs, cudaEvent_t cache_ready, void* stream) {
  if (!m || !c || !cand_offsets) return TXS_ERR_INVALID_ARG;
  if (c->model_hash != m->hash) return TXS_ERR_STALE_CACHE;
  if (n_req != c->n_req || !offsets_ok(cand_offsets, n_req, false)) return TXS_ERR_INVALID_ARG;
  if (n_req > kMaxReqParam) return TXS_ERR_UNSUPPORTED;
  const txs_config& cf = m->cfg;
  const long long n_cand = cand_offsets[n_req];
  if (n_cand + static_cast<long long>(n_req) * cf.n_ctx > 0x7FFFFFFFLL) return TXS_ERR_UNSUPPORTED;
  if (n_cand == 0) return TXS_OK;
  if (!cand_tok || !out_logits || (cf.n_ctx > 0 && !ctx_tok) || !workspace) return TXS_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(workspace) & 255) return TXS_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(cand_tok) & 15) || (ctx_tok && (reinterpret_cast<uintptr_t>(ctx_tok) & 15)))
    return TXS_ERR_INVALID_ARG;
  if (workspace_bytes < score_layout(cf, m->es, n_req, n_cand).total) return TXS_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const KvView v{c->kv, c->cap_total, c->d_off, c->d_len, c->gkv, cache_ready};
  return cf.dtype == TXS_BF16
             ? score_impl<__nv_bfloat16>(m, v, n_req, cand_offsets, cand_tok, ctx_tok, workspace, out_logits,
                                         out_probs, s)
             : score_impl<float>(m, v, n_req, cand_offsets, cand_tok, ctx_tok, workspace, out_logits, out_probs, s);
}
}  // namespace
}  // namespace txs

TXS_API txs_status txs_score_candidates(txs_model* m, const txs_kv_cache* c, int32_t n_req,
                                        const int32_t* cand_offsets, const void* cand_tok, const void* ctx_tok,
                                        void* workspace, size_t workspace_bytes, float* out_logits, float* out_probs,
                                        void* stream) {
  TXS_TRACE();
  return score_entry(m, c, n_req, cand_offsets, cand_tok, ctx_tok, workspace, workspace_bytes, out_logits,
                     out_probs, nullptr, stream);
}

TXS_API txs_status txs_score_candidates_after(txs_model* m, const txs_kv_cache* c, int32_t n_req,
                                              const int32_t* cand_offsets, const void* cand_tok,
                                              const void* ctx_tok, void* workspace, size_t workspace_bytes,
                                              float* out_logits, float* out_probs, void* cache_ready,
                                              void* stream) {
  TXS_TRACE();
  return score_entry(m, c, n_req, cand_offsets, cand_tok, ctx_tok, workspace, workspace_bytes, out_logits,
                     out_probs, static_cast<cudaEvent_t>(cache_ready), stream);
}

// Streaming events: the score workspace, then per event its cache view
// (first row, length), pooled anchor g and the anchor's K/V projections.
struct EventsLayout {
  size_t score, ev_off, ev_len, g, gkv, part, total;
};
EventsLayout events_layout(const txs_config& cf, int es, int n_ev, long long n_cand, int max_end) {
  EventsLayout L;
  size_t o = score_layout(cf, es, n_ev, n_cand).total;
  auto take = [&](size_t bytes) {
    const size_t at = o;
    o += (bytes + 255) / 256 * 256;
    return at;
  };
  L.score = 0;
  L.ev_off = take(sizeof(int) * n_ev);
  L.ev_len = take(sizeof(int) * n_ev);
  L.g = take(sizeof(float) * n_ev * cf.d_model);
  L.gkv = take(sizeof(float) * 2 * cf.n_layers * n_ev * kv_dim(cf));
  L.part = take(sizeof(float) * prefix_pool_scratch_floats(max_end, cf.d_model));
  L.total = o;
  return L;
}

TXS_API txs_status txs_events_workspace_size(const txs_model* m, int32_t n_events, int64_t total_cand,
                                             int32_t max_event_end, size_t* bytes) {
  TXS_TRACE();
  if (!m || !bytes || n_events < 0 || total_cand < 0 || max_event_end < 0) return TXS_ERR_INVALID_ARG;
  *bytes = events_layout(m->cfg, m->es, n_events, total_cand, max_event_end).total;
  return TXS_OK;
}

template <typename T>
txs_status events_impl(txs_model* m, const txs_kv_cache* c, int user, const void* beh_enc, int n_ev,
                       const int32_t* ends, const int32_t* cand_off, const void* cand_tok, const void* ctx_tok,
                       void* ws, float* logits, float* probs, cudaStream_t s) {
  const txs_config& cf = m->cfg;
  const int d = cf.d_model, nL = cf.n_layers;
  int max_end = 0;
  for (int t = 0; t < n_ev; ++t) max_end = std::max(max_end, static_cast<int>(ends[t]));
  const EventsLayout L = events_layout(cf, sizeof(T), n_ev, cand_off[n_ev], max_end);
  uint8_t* base = static_cast<uint8_t*>(ws);
  int* ev_off = reinterpret_cast<int*>(base + L.ev_off);
  int* ev_len = reinterpret_cast<int*>(base + L.ev_len);
  float* g = reinterpret_cast<float*>(base + L.g);
  float* gkv = reinterpret_cast<float*>(base + L.gkv);
  float* part = reinterpret_cast<float*>(base + L.part);
  // per-event anchors pooled over each prefix, projected by every layer's W_K, W_V
  TXS_CK(launch_prefix_pool<T>(static_cast<const T*>(beh_enc), ends, n_ev, c->h_off[user], m->w_pool, d, part, g,
                               ev_off, ev_len, s));
  TXS_CK(launch_anchor_proj<T>(g, static_cast<const T*>(m->Wt_kv), m->b_kv, gkv, n_ev, d, c->dkv, nL, s));
  const KvView v{c->kv, c->cap_total, ev_off, ev_len, gkv};
  return score_impl<T>(m, v, n_ev, cand_off, cand_tok, ctx_tok, ws, logits, probs, s);
}

TXS_API txs_status txs_score_events(txs_model* m, const txs_kv_cache* c, int32_t user, const void* beh_enc,
                                    int32_t n_events, const int32_t* event_ends, const int32_t* cand_offsets,
                                    const void* cand_tok, const void* ctx_tok, void* workspace,
                                    size_t workspace_bytes, float* out_logits, float* out_probs, void* stream) {
  TXS_TRACE();
  if (!m || !c || !event_ends || !cand_offsets || n_events < 0) return TXS_ERR_INVALID_ARG;
  if (c->model_hash != m->hash) return TXS_ERR_STALE_CACHE;
  if (user < 0 || user >= c->n_req) return TXS_ERR_INVALID_ARG;
  if (n_events == 0) return TXS_OK;
  if (n_events > kMaxReqParam) return TXS_ERR_UNSUPPORTED;
  if (!offsets_ok(cand_offsets, n_events, false)) return TXS_ERR_INVALID_ARG;
  for (int t = 0; t < n_events; ++t) {
    if (event_ends[t] == 0) return TXS_ERR_COLD_START;
    if (event_ends[t] < 0 || event_ends[t] > c->h_len[user]) return TXS_ERR_INVALID_ARG;
  }
  const txs_config& cf = m->cfg;
  const long long n_cand = cand_offsets[n_events];
  if (n_cand + static_cast<long long>(n_events) * cf.n_ctx > 0x7FFFFFFFLL) return TXS_ERR_UNSUPPORTED;
  if (n_cand == 0) return TXS_OK;
  if (!beh_enc || !cand_tok || !out_logits || (cf.n_ctx > 0 && !ctx_tok) || !workspace) return TXS_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(workspace) & 255) return TXS_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(cand_tok) & 15) || (ctx_tok && (reinterpret_cast<uintptr_t>(ctx_tok) & 15)) ||
      (reinterpret_cast<uintptr_t>(beh_enc) & 15))
    return TXS_ERR_INVALID_ARG;
  int max_end = 0;
  for (int t = 0; t < n_events; ++t) max_end = std::max(max_end, static_cast<int>(event_ends[t]));
  if (cf.d_model > 512) return TXS_ERR_UNSUPPORTED;
  if (workspace_bytes < events_layout(cf, m->es, n_events, n_cand, max_end).total) return TXS_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  return cf.dtype == TXS_BF16
             ? events_impl<__nv_bfloat16>(m, c, user, beh_enc, n_events, event_ends, cand_offsets, cand_tok, ctx_tok,
                                          workspace, out_logits, out_probs, s)
             : events_impl<float>(m, c, user, beh_enc, n_events, event_ends, cand_offsets, cand_tok, ctx_tok,
                                  workspace, out_logits, out_probs, s);
}

TXS_API txs_status txs_rank_candidates(int32_t n_req, const int32_t* cand_offsets, const float* probs,
                                       int32_t n_actions, int32_t action, int32_t top_k, int32_t* out_idx,
                                       void* stream) {
  TXS_TRACE();
  if (n_req < 0 || !cand_offsets || n_actions < 1 || action < 0 || action >= n_actions || top_k < 0)
    return TXS_ERR_INVALID_ARG;
  if (n_req == 0) return TXS_OK;
  if (!offsets_ok(cand_offsets, n_req, false)) return TXS_ERR_INVALID_ARG;
  if (n_req > kMaxReqParam) return TXS_ERR_UNSUPPORTED;
  for (int r = 0; r < n_req; ++r)
    if (cand_offsets[r + 1] - cand_offsets[r] > 32768) return TXS_ERR_UNSUPPORTED;
  if (cand_offsets[n_req] == 0 && top_k == 0) return TXS_OK;
  if (!out_idx || (!probs && cand_offsets[n_req] > 0)) return TXS_ERR_INVALID_ARG;
  cudaError_t err = launch_rank(n_req, cand_offsets, probs, n_actions, action, top_k, out_idx,
                                static_cast<cudaStream_t>(stream));
  if (err != cudaSuccess) return fail_cuda("rank", err);
  return TXS_OK;
}

TXS_API txs_status txs_device_status(txs_model* m) {
  TXS_TRACE();
  if (!m) return TXS_ERR_INVALID_ARG;
  cudaError_t err = cudaDeviceSynchronize();
  if (err != cudaSuccess) return fail_cuda("cudaDeviceSynchronize", err);
  int v = 0;
  if ((err = cudaMemcpy(&v, m->status, 4, cudaMemcpyDeviceToHost)) != cudaSuccess) return fail_cuda("status", err);
  if (v != 0 && (err = cudaMemset(m->status, 0, 4)) != cudaSuccess) return fail_cuda("status reset", err);
  return static_cast<txs_status>(v);
}

TXS_API txs_status txs_selftest_wait_timeout(txs_model* m, void* stream) {
  TXS_TRACE();
  if (!m) return TXS_ERR_INVALID_ARG;
  const cudaError_t e = launch_wait_timeout_probe(m->status, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? TXS_OK : fail_cuda("wait_timeout_probe", e);
}

TXS_API txs_status txs_gelu_eval(const float* x, float* y, int64_t n, int32_t variant, void* stream) {
  TXS_TRACE();
  if (n < 0 || (n > 0 && (!x || !y)) || (variant != 0 && variant != 1)) return TXS_ERR_INVALID_ARG;
  const cudaError_t e = launch_gelu_eval(x, y, n, variant, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? TXS_OK : fail_cuda("gelu_eval", e);
}

TXS_API txs_status txs_profile_enable(int32_t enable) {
  TXS_TRACE();
  g_prof.on = enable != 0;
  return TXS_OK;
}

TXS_API txs_status txs_profile_collect(double* total_ms, int64_t* launches, int32_t n) {
  TXS_TRACE();
  if (!total_ms || !launches || n < TXS_N_KERNEL_CLASSES) return TXS_ERR_INVALID_ARG;
  for (int i = 0; i < n; ++i) {
    total_ms[i] = 0;
    launches[i] = 0;
  }
  txs_status st = TXS_OK;
  for (ProfRec& r : g_prof.recs) {
    float ms = 0.f;
    if (cudaEventSynchronize(r.b) != cudaSuccess || cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess)
      st = TXS_ERR_CUDA;
    total_ms[r.cls] += ms;
    launches[r.cls] += 1;
    g_prof.pool.push_back(r.a);
    g_prof.pool.push_back(r.b);
  }
  g_prof.recs.clear();
  return st;
}

TXS_API const char* txs_kernel_class_name(int32_t cls) {
  TXS_TRACE();
  static const char* names[] = {"pack", "gemm_qkv", "attn_serving", "gemm_oproj_ln", "gemm_q", "attn_cross",
                                "gemm_ffn1_gelu", "gemm_ffn2_ln", "gemm_kv_build", "pool", "global_kv", "rank",
                                "misc", "row_ln", "cand_mlp", "enc_embed", "enc_gemm", "enc_attn", "head_dw",
                                "gemm_q_attn_lg"};
  if (cls < 0 || cls >= KC_COUNT_) return "";
  return names[cls];
}
