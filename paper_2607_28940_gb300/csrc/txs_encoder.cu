// C ABI of the behavior-stream encoder (Sec. 4.1.1) and its incremental
// update (App. D, incremental-encoding remark): host-side validation, handle
// and state management, and the order of launches of one encode call.  The
// arithmetic runs in k_encoder.cu (token embedding, causal relative-bias
// attention) and on the library's GEMMs (projections, FFN, residual + LN
// epilogues).
#include <algorithm>
#include <cmath>
#include <cstring>
#include <string>
#include <type_traits>
#include <vector>

#include "txs_internal.cuh"

namespace txs {
struct EncLayerW {
  void *Wt_qkv, *Wt_o, *Wt_1, *Wt_2;  // transposed weights [d_out, d_in]
  float *b_qkv, *b_o, *g1, *be1, *b_1, *b_2, *g2, *be2;
};
}  // namespace txs

struct txs_encoder {
  txs_enc_config cfg;
  int es = 0;
  std::vector<void*> allocs;
  std::vector<txs::EncLayerW> layers;
  float* rel = nullptr;     // [nL][H][R] relative bias * log2(e)
  void* E_type = nullptr;   // [n_types, type_dim] config dtype
  int* status = nullptr;
  uint64_t hash = 0;
};

struct txs_enc_state {
  int n_req = 0, n_layers = 0, d = 0, es = 0;
  uint64_t enc_hash = 0;
  long long cap_total = 0;
  std::vector<int> h_off, h_len;     // slot offsets [R+1], token counts [R]
  int* d_off = nullptr;              // [R+1]
  int* d_call = nullptr;             // [3R+2]: in_off [R+1] | dst0 [R] | tile_off [R+1]
  void* kv = nullptr;                // [nL][2][cap_total][d]
  int* h_stage = nullptr;            // pinned ring of 4 upload slots
  int stage_ints = 0, stage_next = 0;
  cudaEvent_t stage_ev[4] = {nullptr, nullptr, nullptr, nullptr};
  std::vector<void*> allocs;
};

namespace txs {
namespace {

txs_status enc_fail(const char* where, cudaError_t e) {
  set_last_error((std::string(where) + ": " + cudaGetErrorString(e)).c_str());
  return TXS_ERR_CUDA;
}

#define ENC_CK(call)                                   \
  do {                                                 \
    cudaError_t e_ = (call);                           \
    if (e_ != cudaSuccess) return enc_fail(#call, e_); \
  } while (0)

bool enc_cfg_ok(const txs_enc_config& c, std::string* why) {
  auto bad = [&](const char* m) {
    *why = m;
    return false;
  };
  if (c.dtype != TXS_FP32 && c.dtype != TXS_BF16) return bad("dtype");
  if (c.n_layers < 1 || c.n_layers > 16) return bad("n_layers");
  if (c.n_heads < 1 || c.d_model % c.n_heads) return bad("n_heads");
  const int dh = c.d_model / c.n_heads;
  if (dh != 32 && dh != 64) return bad("d_head must be 32 or 64");
  if (c.dtype == TXS_BF16) {
    if (c.d_model != 64 && c.d_model != 128 && c.d_model != 256 && c.d_model != 512) return bad("d_model (bf16)");
  } else if (c.d_model % 32 || c.d_model > 512 || c.d_model < 32) {
    return bad("d_model (fp32)");
  }
  if (c.d_ff < 64 || c.d_ff % 64 || c.d_ff > 16384) return bad("d_ff");
  if (c.type_dim < 0 || c.type_dim >= c.d_model) return bad("type_dim");
  if (c.type_dim > 0 && c.n_types < 1) return bad("n_types");
  if (c.n_rel < 1 || c.n_rel > 65536) return bad("n_rel");
  if (c.window < 0) return bad("window");
  if (!(c.ln_eps > 0.f) || !std::isfinite(c.ln_eps)) return bad("ln_eps");
  if (c.dtype == TXS_BF16) {
    const int d = c.d_model, F = c.d_ff;
    if (!tc_gemm_supported(d, d, EPI_BIAS) || !tc_gemm_supported(2 * d, d, EPI_KV) ||
        !tc_gemm_supported(d, d, EPI_LN) || !tc_gemm_supported(F, d, EPI_BIAS_GELU) ||
        !tc_gemm_supported(d, F, EPI_LN))
      return bad("GEMM shape");
  }
  return true;
}

void* enc_alloc(std::vector<void*>& list, size_t bytes, cudaError_t* err) {
  void* p = nullptr;
  *err = cudaMalloc(&p, bytes ? bytes : 16);
  if (*err != cudaSuccess) return nullptr;
  list.push_back(p);
  return p;
}

size_t al256(size_t x) { return (x + 255) & ~size_t(255); }

struct EncWs {
  size_t X, Q, A, H1, Hf, tmp, total;
};

EncWs enc_ws_layout(const txs_enc_config& c, int es, long long n) {
  const size_t d = c.d_model, F = c.d_ff;
  EncWs L{};
  size_t o = 0;
  auto take = [&](size_t b) {
    size_t at = o;
    o = al256(o + b);
    return at;
  };
  L.X = take(n * d * es);
  L.Q = take(n * d * es);
  L.A = take(n * d * es);
  L.H1 = take(n * d * es);
  L.Hf = take(n * F * es);
  L.tmp = take(c.dtype == TXS_FP32 ? n * d * 4 : 0);
  L.total = o;
  return L;
}

cudaError_t enc_gemm(const txs_encoder* m, const void* A, long long lda, const void* Bt, EpiArgs e, float* tmp,
                     cudaStream_t s) {
  e.status = m->status;
  if (m->cfg.dtype == TXS_BF16)
    return launch_gemm_tc(static_cast<const __nv_bfloat16*>(A), lda, static_cast<const __nv_bfloat16*>(Bt), e, s,
                          KC_ENC_GEMM);
  return launch_gemm_simt<float>(static_cast<const float*>(A), lda, static_cast<const float*>(Bt), e, tmp, s,
                                 KC_ENC_GEMM);
}

EpiArgs enc_epi(int epi, long long M, int N, int K) {
  EpiArgs e;
  std::memset(&e, 0, sizeof(e));
  e.epi = epi;
  e.M = static_cast<int>(M);
  e.N = N;
  e.K = K;
  return e;
}

template <typename T>
txs_status enc_prepare(txs_encoder* m, const void* const* w, cudaStream_t s) {
  const txs_enc_config& c = m->cfg;
  const int d = c.d_model, F = c.d_ff, nL = c.n_layers, H = c.n_heads, R = c.n_rel;
  cudaError_t err;
  auto wt = [&](int rows, int cols) { return static_cast<T*>(enc_alloc(m->allocs, size_t(rows) * cols * sizeof(T), &err)); };
  auto vf = [&](size_t n) { return static_cast<float*>(enc_alloc(m->allocs, n * 4, &err)); };
  auto W = [&](int l, int i) { return static_cast<const T*>(w[l * TXS_ENC_WEIGHTS_PER_LAYER + i]); };
  if (!(m->rel = vf(size_t(nL) * H * R))) return enc_fail("cudaMalloc", err);
  for (int l = 0; l < nL; ++l) {
    EncLayerW L;
    T* p;
    if (!(p = wt(3 * d, d))) return enc_fail("cudaMalloc", err);
    ENC_CK(launch_transpose<T>(W(l, 0), p, d, 3 * d, s));
    L.Wt_qkv = p;
    if (!(p = wt(d, d))) return enc_fail("cudaMalloc", err);
    ENC_CK(launch_transpose<T>(W(l, 3), p, d, d, s));
    L.Wt_o = p;
    if (!(p = wt(F, d))) return enc_fail("cudaMalloc", err);
    ENC_CK(launch_transpose<T>(W(l, 7), p, d, F, s));
    L.Wt_1 = p;
    if (!(p = wt(d, F))) return enc_fail("cudaMalloc", err);
    ENC_CK(launch_transpose<T>(W(l, 9), p, F, d, s));
    L.Wt_2 = p;
    float** dst[] = {&L.b_qkv, &L.b_o, &L.g1, &L.be1, &L.b_1, &L.b_2, &L.g2, &L.be2};
    const int idx[] = {1, 4, 5, 6, 8, 10, 11, 12};
    const int len[] = {3 * d, d, d, d, F, d, d, d};
    for (int i = 0; i < 8; ++i) {
      float* v = vf(len[i]);
      if (!v) return enc_fail("cudaMalloc", err);
      ENC_CK(launch_to_f32<T>(W(l, idx[i]), v, len[i], s));
      *dst[i] = v;
    }
    ENC_CK(launch_enc_rel_prep<T>(W(l, 2), m->rel + size_t(l) * H * R, H * R, s));
    m->layers.push_back(L);
  }
  const void* const* tail = w + nL * TXS_ENC_WEIGHTS_PER_LAYER;
  const size_t ntype = c.type_dim ? size_t(c.n_types) * c.type_dim : 0;
  if (ntype) {
    if (!(m->E_type = enc_alloc(m->allocs, ntype * sizeof(T), &err))) return enc_fail("cudaMalloc", err);
    ENC_CK(cudaMemcpyAsync(m->E_type, tail[0], ntype * sizeof(T), cudaMemcpyDeviceToDevice, s));
  }
  // content hash of the config and every weight tensor
  unsigned long long* dh = static_cast<unsigned long long*>(enc_alloc(m->allocs, 8, &err));
  if (!dh) return enc_fail("cudaMalloc", err);
  ENC_CK(cudaMemsetAsync(dh, 0, 8, s));
  const size_t es = sizeof(T);
  for (int l = 0; l < nL; ++l) {
    const size_t n[TXS_ENC_WEIGHTS_PER_LAYER] = {size_t(d) * 3 * d, 3 * size_t(d), size_t(H) * R, size_t(d) * d,
                                                 size_t(d), size_t(d), size_t(d), size_t(d) * F, size_t(F),
                                                 size_t(F) * d, size_t(d), size_t(d), size_t(d)};
    for (int i = 0; i < TXS_ENC_WEIGHTS_PER_LAYER; ++i)
      ENC_CK(launch_hash(W(l, i), static_cast<long long>(n[i] * es), 300000 + uint64_t(l) * 64 + i, dh, s));
  }
  if (ntype) ENC_CK(launch_hash(tail[0], static_cast<long long>(ntype * es), 400000, dh, s));
  unsigned long long hv = 0;
  ENC_CK(cudaMemcpyAsync(&hv, dh, 8, cudaMemcpyDeviceToHost, s));
  ENC_CK(cudaStreamSynchronize(s));
  uint64_t h = hv ^ 0x656E636F64657231ull;
  const int32_t cf[] = {c.d_model, c.n_heads, c.d_ff, c.n_layers, c.type_dim, c.n_types, c.n_rel, c.window, c.dtype};
  for (int32_t v : cf) h = (h ^ static_cast<uint64_t>(static_cast<uint32_t>(v))) * 0x100000001B3ull;
  uint32_t eps_bits;
  std::memcpy(&eps_bits, &c.ln_eps, 4);
  m->hash = (h ^ eps_bits) * 0x100000001B3ull;
  return TXS_OK;
}

// Upload n ints through the state's pinned ring (a slot is reused only after
// the copy that last read it has run).
cudaError_t enc_upload(txs_enc_state* st, int* dst, const int* src, int n, cudaStream_t s) {
  const int i = st->stage_next;
  st->stage_next = (i + 1) & 3;
  cudaEventSynchronize(st->stage_ev[i]);
  int* slot = st->h_stage + static_cast<size_t>(i) * st->stage_ints;
  std::memcpy(slot, src, sizeof(int) * n);
  cudaError_t err = cudaMemcpyAsync(dst, slot, sizeof(int) * n, cudaMemcpyHostToDevice, s);
  if (err != cudaSuccess) return err;
  return cudaEventRecord(st->stage_ev[i], s);
}

// One encode call: user r's rows in_off[r] .. in_off[r+1] go after its
// current tokens (append) or from position 0 (build).
template <typename T>
txs_status encode_impl(txs_encoder* m, txs_enc_state* st, const int32_t* in_off, const void* subj,
                       const int32_t* types, void* ws, void* phi_out, bool append, cudaStream_t s) {
  const txs_enc_config& c = m->cfg;
  const int R = st->n_req, d = c.d_model, F = c.d_ff, H = c.n_heads;
  const long long n = in_off[R];
  int max_new = 0;
  for (int r = 0; r < R; ++r) max_new = std::max(max_new, in_off[r + 1] - in_off[r]);
  // bf16: tensor-core attention (128-row tiles) for build and append alike,
  // which keeps incremental encoding bit-identical to a full encode
  const bool use_tc = std::is_same<T, __nv_bfloat16>::value && enc_attn_tc_supported(d, H, c.n_rel);
  const int QT = use_tc ? 128 : enc_query_tile(max_new);
  std::vector<int> up(3 * R + 2);
  int tiles = 0;
  for (int r = 0; r <= R; ++r) up[r] = in_off[r];
  for (int r = 0; r < R; ++r) up[R + 1 + r] = st->h_off[r] + (append ? st->h_len[r] : 0);
  for (int r = 0; r < R; ++r) {
    up[2 * R + 1 + r] = tiles;
    tiles += (in_off[r + 1] - in_off[r] + QT - 1) / QT;
  }
  up[3 * R + 1] = tiles;
  if (n == 0) return TXS_OK;
  {
    // kernel parameters when they fit (capturable), else the pinned ring
    cudaError_t err = launch_upload_ints(st->d_call, up.data(), 3 * R + 2, nullptr, nullptr, 0, s);
    if (err == cudaErrorNotSupported) err = enc_upload(st, st->d_call, up.data(), 3 * R + 2, s);
    if (err != cudaSuccess) return enc_fail("upload", err);
  }
  const int* d_in_off = st->d_call;
  const int* d_dst0 = st->d_call + R + 1;
  const int* d_tile_off = st->d_call + 2 * R + 1;

  const EncWs L = enc_ws_layout(c, sizeof(T), n);
  uint8_t* base = static_cast<uint8_t*>(ws);
  T* X = reinterpret_cast<T*>(base + L.X);
  T* Q = reinterpret_cast<T*>(base + L.Q);
  T* A = reinterpret_cast<T*>(base + L.A);
  T* H1 = reinterpret_cast<T*>(base + L.H1);
  T* Hf = reinterpret_cast<T*>(base + L.Hf);
  float* tmp = reinterpret_cast<float*>(base + L.tmp);

  ENC_CK(launch_enc_embed<T>(static_cast<const T*>(subj), types, static_cast<const T*>(m->E_type), X, n, d,
                             c.type_dim, c.n_types, m->status, s));
  T* kv = static_cast<T*>(st->kv);
  for (int l = 0; l < c.n_layers; ++l) {
    const EncLayerW& W = m->layers[l];
    T* Kl = kv + size_t(2 * l) * st->cap_total * d;
    T* Vl = Kl + size_t(st->cap_total) * d;
    // q = X W_q + b_q; the new rows' k, v go straight into their cache slots
    EpiArgs e = enc_epi(EPI_BIAS, n, d, d);
    e.bias = W.b_qkv;
    e.out = Q;
    e.ldo = d;
    ENC_CK(enc_gemm(m, X, d, W.Wt_qkv, e, tmp, s));
    e = enc_epi(EPI_KV, n, 2 * d, d);
    e.bias = W.b_qkv + d;
    e.out = Kl;
    e.ldo = d;
    e.seg_off = d_in_off;
    e.dst_row0 = d_dst0;
    e.n_seg = R;
    e.col_blk = d;
    e.col_blk_stride = st->cap_total * d;
    ENC_CK(enc_gemm(m, X, d, static_cast<const T*>(W.Wt_qkv) + size_t(d) * d, e, tmp, s));
    // causal attention with the relative position bias
    const float* beta = m->rel + size_t(l) * H * c.n_rel;
    if constexpr (std::is_same<T, __nv_bfloat16>::value) {
      if (use_tc) {
        ENC_CK(launch_enc_attn_tc(Q, Kl, Vl, A, st->cap_total, d_in_off, d_dst0, st->d_off, d_tile_off, R, tiles,
                                  beta, c.n_rel, c.window, H, d, m->status, s));
      } else {
        ENC_CK(launch_enc_attn<T>(Q, Kl, Vl, A, d_in_off, d_dst0, st->d_off, d_tile_off, R, tiles, QT, beta,
                                  c.n_rel, c.window, H, d, m->status, s));
      }
    } else {
      ENC_CK(launch_enc_attn<T>(Q, Kl, Vl, A, d_in_off, d_dst0, st->d_off, d_tile_off, R, tiles, QT, beta,
                                c.n_rel, c.window, H, d, m->status, s));
    }
    // H = LN1(X + A W_o + b_o)
    e = enc_epi(EPI_LN, n, d, d);
    e.bias = W.b_o;
    e.res = X;
    e.ldr = d;
    e.gamma = W.g1;
    e.beta = W.be1;
    e.ln_eps = c.ln_eps;
    e.out = H1;
    e.ldo = d;
    ENC_CK(enc_gemm(m, A, d, W.Wt_o, e, tmp, s));
    // Y = LN2(H + GELU(H W_1 + b_1) W_2 + b_2): the next layer's input, or Phi_b
    e = enc_epi(EPI_BIAS_GELU, n, F, d);
    e.bias = W.b_1;
    e.out = Hf;
    e.ldo = F;
    ENC_CK(enc_gemm(m, H1, d, W.Wt_1, e, tmp, s));
    e = enc_epi(EPI_LN, n, d, F);
    e.bias = W.b_2;
    e.res = H1;
    e.ldr = d;
    e.gamma = W.g2;
    e.beta = W.be2;
    e.ln_eps = c.ln_eps;
    e.out = l == c.n_layers - 1 ? phi_out : static_cast<void*>(X);
    e.ldo = d;
    ENC_CK(enc_gemm(m, Hf, F, W.Wt_2, e, tmp, s));
  }
  return TXS_OK;
}

bool offsets_nondecreasing(const int32_t* off, int n) {
  if (!off || off[0] != 0) return false;
  for (int i = 0; i < n; ++i)
    if (off[i + 1] < off[i]) return false;
  return true;
}

void state_free(txs_enc_state* st) {
  if (!st) return;
  for (void* p : st->allocs) cudaFree(p);
  for (cudaEvent_t& e : st->stage_ev)
    if (e) cudaEventDestroy(e);
  if (st->h_stage) cudaFreeHost(st->h_stage);
  delete st;
}

}  // namespace
}  // namespace txs

using namespace txs;

TXS_API txs_status txs_encoder_create(const txs_enc_config* cfg, const void* const* weights, txs_encoder** out) {
  TXS_TRACE();
  if (!cfg || !weights || !out) return TXS_ERR_INVALID_ARG;
  *out = nullptr;
  std::string why;
  if (!enc_cfg_ok(*cfg, &why)) {
    set_last_error(why.c_str());
    return cfg->dtype != TXS_FP32 && cfg->dtype != TXS_BF16 ? TXS_ERR_INVALID_ARG : TXS_ERR_UNSUPPORTED;
  }
  const int nw = cfg->n_layers * TXS_ENC_WEIGHTS_PER_LAYER + (cfg->type_dim ? 1 : 0);
  for (int i = 0; i < nw; ++i)
    if (!weights[i]) return TXS_ERR_INVALID_ARG;
  cudaError_t err = cudaDeviceSynchronize();
  if (err != cudaSuccess) return enc_fail("cudaDeviceSynchronize", err);
  txs_encoder* m = new txs_encoder();
  m->cfg = *cfg;
  m->es = cfg->dtype == TXS_BF16 ? 2 : 4;
  m->status = static_cast<int*>(enc_alloc(m->allocs, 4, &err));
  txs_status st = m->status ? TXS_OK : enc_fail("cudaMalloc", err);
  cudaStream_t s = nullptr;
  if (st == TXS_OK && (err = cudaMemset(m->status, 0, 4)) != cudaSuccess) st = enc_fail("cudaMemset", err);
  if (st == TXS_OK)
    st = cfg->dtype == TXS_BF16 ? enc_prepare<__nv_bfloat16>(m, weights, s) : enc_prepare<float>(m, weights, s);
  if (st == TXS_OK && (err = cudaDeviceSynchronize()) != cudaSuccess) st = enc_fail("cudaDeviceSynchronize", err);
  if (st != TXS_OK) {
    cudaDeviceSynchronize();
    txs_encoder_destroy(m);
    return st;
  }
  *out = m;
  return TXS_OK;
}

TXS_API void txs_encoder_destroy(txs_encoder* m) {
  TXS_TRACE();
  if (!m) return;
  for (void* p : m->allocs) cudaFree(p);
  delete m;
}

TXS_API uint64_t txs_encoder_hash(const txs_encoder* m) { return m ? m->hash : 0; }

TXS_API txs_status txs_encoder_workspace_size(const txs_encoder* m, int64_t n_rows, size_t* bytes) {
  TXS_TRACE();
  if (!m || !bytes || n_rows < 0) return TXS_ERR_INVALID_ARG;
  *bytes = enc_ws_layout(m->cfg, m->es, n_rows).total;
  return TXS_OK;
}

namespace txs {
namespace {
// Arguments shared by build and append, checked before anything is enqueued.
txs_status check_call(const txs_encoder* m, int n_req, const int32_t* off, const void* subj, const int32_t* types,
                      void* ws, size_t ws_bytes, void* phi_out) {
  if (!offsets_nondecreasing(off, n_req)) return TXS_ERR_INVALID_ARG;
  const long long n = off[n_req];
  if (n == 0) return TXS_OK;
  if (!subj || !phi_out || !ws || (m->cfg.type_dim > 0 && !types)) return TXS_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(ws) & 255) return TXS_ERR_INVALID_ARG;
  if (ws_bytes < enc_ws_layout(m->cfg, m->es, n).total) return TXS_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(subj) | reinterpret_cast<uintptr_t>(phi_out)) & 15) return TXS_ERR_INVALID_ARG;
  return TXS_OK;
}
}  // namespace
}  // namespace txs

TXS_API txs_status txs_encode_build(txs_encoder* m, int32_t n_req, const int32_t* offsets, const void* subj,
                                    const int32_t* types, int32_t capacity_extra, void* workspace,
                                    size_t workspace_bytes, void* phi_out, void* stream, txs_enc_state** out) {
  TXS_TRACE();
  if (!m || !out || n_req < 1 || capacity_extra < 0 || !offsets) return TXS_ERR_INVALID_ARG;
  *out = nullptr;
  txs_status chk = check_call(m, n_req, offsets, subj, types, workspace, workspace_bytes, phi_out);
  if (chk != TXS_OK) return chk;
  const txs_enc_config& c = m->cfg;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  txs_enc_state* st = new txs_enc_state();
  st->n_req = n_req;
  st->n_layers = c.n_layers;
  st->d = c.d_model;
  st->es = m->es;
  st->enc_hash = m->hash;
  st->h_off.assign(n_req + 1, 0);
  st->h_len.assign(n_req, 0);
  long long tot = 0;
  for (int r = 0; r < n_req; ++r) {
    st->h_off[r] = static_cast<int>(tot);
    tot += static_cast<long long>(offsets[r + 1] - offsets[r]) + capacity_extra;
    if (tot > 0x7FFFFFFFLL) {
      delete st;
      return TXS_ERR_UNSUPPORTED;
    }
  }
  st->h_off[n_req] = static_cast<int>(tot);
  st->cap_total = tot;
  cudaError_t err = cudaSuccess;
  txs_status rc = TXS_OK;
  auto A = [&](size_t bytes) -> void* {
    if (rc != TXS_OK) return nullptr;
    void* p = enc_alloc(st->allocs, bytes, &err);
    if (!p) rc = enc_fail("cudaMalloc", err);
    return p;
  };
  st->kv = A(size_t(c.n_layers) * 2 * tot * c.d_model * m->es);
  // zeroed: attention tiles may read key rows past a user's tokens (masked,
  // P = 0), which must hold finite values
  if (rc == TXS_OK && (err = cudaMemsetAsync(st->kv, 0, size_t(c.n_layers) * 2 * tot * c.d_model * m->es, s)) !=
                          cudaSuccess)
    rc = enc_fail("cudaMemsetAsync", err);
  st->d_off = static_cast<int*>(A(4 * size_t(n_req + 1)));
  st->d_call = static_cast<int*>(A(4 * size_t(3 * n_req + 2)));
  if (rc == TXS_OK) {
    st->stage_ints = 3 * n_req + 2;
    if ((err = cudaMallocHost(&st->h_stage, sizeof(int) * 4 * st->stage_ints)) != cudaSuccess) {
      st->h_stage = nullptr;
      rc = enc_fail("cudaMallocHost", err);
    }
    for (int i = 0; i < 4 && rc == TXS_OK; ++i)
      if ((err = cudaEventCreateWithFlags(&st->stage_ev[i], cudaEventDisableTiming)) != cudaSuccess)
        rc = enc_fail("cudaEventCreate", err);
  }
  if (rc == TXS_OK && (err = enc_upload(st, st->d_off, st->h_off.data(), n_req + 1, s)) != cudaSuccess)
    rc = enc_fail("upload", err);
  if (rc == TXS_OK)
    rc = c.dtype == TXS_BF16
             ? encode_impl<__nv_bfloat16>(m, st, offsets, subj, types, workspace, phi_out, false, s)
             : encode_impl<float>(m, st, offsets, subj, types, workspace, phi_out, false, s);
  if (rc != TXS_OK) {
    cudaStreamSynchronize(s);
    state_free(st);
    return rc;
  }
  for (int r = 0; r < n_req; ++r) st->h_len[r] = offsets[r + 1] - offsets[r];
  *out = st;
  return TXS_OK;
}

TXS_API txs_status txs_encode_append(txs_encoder* m, txs_enc_state* st, int32_t n_req, const int32_t* new_offsets,
                                     const void* subj, const int32_t* types, void* workspace,
                                     size_t workspace_bytes, void* phi_out, void* stream) {
  TXS_TRACE();
  if (!m || !st || !new_offsets) return TXS_ERR_INVALID_ARG;
  if (n_req != st->n_req) return TXS_ERR_INVALID_ARG;
  if (st->enc_hash != m->hash) return TXS_ERR_STALE_CACHE;
  txs_status chk = check_call(m, n_req, new_offsets, subj, types, workspace, workspace_bytes, phi_out);
  if (chk != TXS_OK) return chk;
  for (int r = 0; r < n_req; ++r)
    if (static_cast<long long>(st->h_len[r]) + (new_offsets[r + 1] - new_offsets[r]) >
        st->h_off[r + 1] - st->h_off[r])
      return TXS_ERR_CAPACITY;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const txs_status rc =
      m->cfg.dtype == TXS_BF16
          ? encode_impl<__nv_bfloat16>(m, st, new_offsets, subj, types, workspace, phi_out, true, s)
          : encode_impl<float>(m, st, new_offsets, subj, types, workspace, phi_out, true, s);
  if (rc != TXS_OK) return rc;
  for (int r = 0; r < n_req; ++r) st->h_len[r] += new_offsets[r + 1] - new_offsets[r];
  return TXS_OK;
}

TXS_API txs_status txs_enc_state_lengths(const txs_enc_state* st, int32_t* out_len) {
  TXS_TRACE();
  if (!st || !out_len) return TXS_ERR_INVALID_ARG;
  std::copy(st->h_len.begin(), st->h_len.end(), out_len);
  return TXS_OK;
}

TXS_API int32_t txs_enc_state_n_req(const txs_enc_state* st) { return st ? st->n_req : 0; }

TXS_API txs_status txs_enc_state_read_rows(const txs_enc_state* st, int32_t layer, int32_t which, int32_t req,
                                           int32_t row0, int32_t n_rows, void* dst, void* stream) {
  TXS_TRACE();
  if (!st || !dst || layer < 0 || layer >= st->n_layers || which < 0 || which > 1 || req < 0 || req >= st->n_req ||
      row0 < 0 || n_rows < 0 || static_cast<long long>(row0) + n_rows > st->h_len[req])
    return TXS_ERR_INVALID_ARG;
  if (n_rows == 0) return TXS_OK;
  const size_t row_bytes = size_t(st->d) * st->es;
  const size_t at = (size_t(2 * layer + which) * st->cap_total + st->h_off[req] + row0) * row_bytes;
  cudaError_t err = cudaMemcpyAsync(dst, static_cast<const uint8_t*>(st->kv) + at, n_rows * row_bytes,
                                    cudaMemcpyDeviceToDevice, static_cast<cudaStream_t>(stream));
  if (err != cudaSuccess) return enc_fail("cudaMemcpyAsync", err);
  return TXS_OK;
}

TXS_API void txs_enc_state_destroy(txs_enc_state* st) {
  TXS_TRACE();
  if (!st) return;
  cudaDeviceSynchronize();
  state_free(st);
}

TXS_API txs_status txs_encoder_device_status(txs_encoder* m) {
  TXS_TRACE();
  if (!m) return TXS_ERR_INVALID_ARG;
  cudaError_t err = cudaDeviceSynchronize();
  if (err != cudaSuccess) return enc_fail("cudaDeviceSynchronize", err);
  int v = 0;
  if ((err = cudaMemcpy(&v, m->status, 4, cudaMemcpyDeviceToHost)) != cudaSuccess) return enc_fail("status", err);
  if (v != 0 && (err = cudaMemset(m->status, 0, 4)) != cudaSuccess) return enc_fail("status reset", err);
  return static_cast<txs_status>(v);
}
