// Attention on the tensor cores (tcgen05, TMA, TMEM):
//   fa_pair_kernel  multi-query cross-attention over all cached rows of a
//                   request (FULL key set: the -sparseAttn variant of
//                   Sec. 5.2; sparse cross-attention equation of Sec. 4.1.2
//                   with I = every behavior row);
//   enc_fa_kernel   causal self-attention of the behavior encoder with a
//                   relative position bias (Sec. 4.1.1, App. D).
// Both follow one pipeline.  All query rows of a request (or of a user)
// share its K/V (Sec. 4.1.2 multi-query formulation), so each 128-key K/V
// tile is staged once per CTA and serves every query row of the CTA:
//   warp 0     TMA producer: K_j, V_j tiles (one head's columns) into a
//              STG-deep shared-memory ring;
//   warp 1     MMA issuer: S_j = Q K_j^T into TMEM, then O += P_j V_j into
//              the TMEM output tile.  Q and P are the A operands and are read
//              from TMEM, so the tensor core reads only K and V from shared
//              memory (V used MN-major: no transpose);
//   softmax    one query row per thread straight out of TMEM (row max,
//              exp2, row sum need no shuffles); P_j (bf16) goes back to TMEM.
// The running maximum is raised only when a tile's maximum exceeds it by more
// than 2^8 (then O and the row sum are rescaled in place); otherwise the
// stale maximum is kept, P stays below 256 and no rescale is needed.  Exact
// softmax is recovered at the end from O / l either way.
// All waits are bounded; a timeout latches TXS_ERR_DEVICE_TIMEOUT.
#include <algorithm>

#include "tc_ptx.cuh"

namespace txs {
namespace fa {

using namespace tc;

constexpr int BQ = 128;            // queries per CTA (TMEM lanes)
constexpr int BKV = 128;           // keys per K/V tile
constexpr int STG = 4;             // K/V ring depth
constexpr int NUM_THREADS = 192;   // producer, MMA, 4 softmax warps
constexpr float kRescaleLog2 = 8.f;  // raise the running max only past this (log2 units)

// ------------------------------------------------------------------ PTX wrappers
//
// The common tcgen05 / TMA / mbarrier wrappers come from tc_ptx.cuh; the
// attention's waits poll without the suspend-time hint (mbar_wait<false>).
// Below: the TMEM-operand MMA and the wider TMEM loads only this file uses.

// Same, with the A operand (M x 16 bf16, K-major: lane = row, two elements
// per 32-bit column) read from TMEM at a_tmem.
__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// 16 columns of this warp's 32 lanes; completion is awaited by tmem_wait_st.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
      "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
      : "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// 128 consecutive columns of this warp's 32 lanes: one load, one wait.
__device__ __forceinline__ void tmem_ld128(uint32_t taddr, float* v) {
  uint32_t r[128];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x128.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63,%64,%65,%66,%67,%68,%69,%70,%71,%72,%73,%74,%75,%76,%77,%78,%79,%80,%81,%82,%83,%84,%85,%86,%87,%88,%89,%90,%91,%92,%93,%94,%95,%96,%97,%98,%99,%100,%101,%102,%103,%104,%105,%106,%107,%108,%109,%110,%111,%112,%113,%114,%115,%116,%117,%118,%119,%120,%121,%122,%123,%124,%125,%126,%127}, [%128];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]), "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]), "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63]), "=r"(r[64]), "=r"(r[65]), "=r"(r[66]), "=r"(r[67]), "=r"(r[68]), "=r"(r[69]), "=r"(r[70]), "=r"(r[71]), "=r"(r[72]), "=r"(r[73]), "=r"(r[74]), "=r"(r[75]), "=r"(r[76]), "=r"(r[77]), "=r"(r[78]), "=r"(r[79]), "=r"(r[80]), "=r"(r[81]), "=r"(r[82]), "=r"(r[83]), "=r"(r[84]), "=r"(r[85]), "=r"(r[86]), "=r"(r[87]), "=r"(r[88]), "=r"(r[89]), "=r"(r[90]), "=r"(r[91]), "=r"(r[92]), "=r"(r[93]), "=r"(r[94]), "=r"(r[95]), "=r"(r[96]), "=r"(r[97]), "=r"(r[98]), "=r"(r[99]), "=r"(r[100]), "=r"(r[101]), "=r"(r[102]), "=r"(r[103]), "=r"(r[104]), "=r"(r[105]), "=r"(r[106]), "=r"(r[107]), "=r"(r[108]), "=r"(r[109]), "=r"(r[110]), "=r"(r[111]), "=r"(r[112]), "=r"(r[113]), "=r"(r[114]), "=r"(r[115]), "=r"(r[116]), "=r"(r[117]), "=r"(r[118]), "=r"(r[119]), "=r"(r[120]), "=r"(r[121]), "=r"(r[122]), "=r"(r[123]), "=r"(r[124]), "=r"(r[125]), "=r"(r[126]), "=r"(r[127])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 128; ++i) v[i] = __uint_as_float(r[i]);
}

// 2^x on the special-function unit (PTX ex2.approx, flush-to-zero).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Shared-memory matrix descriptor (tcgen05): start address, leading/stride
// byte offsets, descriptor version 1, layout code (2 = 128-byte swizzle,
// 4 = 64-byte swizzle).
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo, uint32_t layout) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
  d |= 1ull << 46;
  d |= static_cast<uint64_t>(layout) << 61;
  return d;
}

// kind::f16 instruction descriptor: D fp32, A/B bf16, A K-major; B K-major or
// MN-major (bit 16).
__host__ __device__ constexpr uint32_t idesc_bf16(int m, int n, bool b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (b_mn_major ? (1u << 16) : 0u) |
         (static_cast<uint32_t>(n >> 3) << 17) | (static_cast<uint32_t>(m >> 4) << 24);
}

// ------------------------------------------------------------------ kernel

struct FaArgs {
  const __nv_bfloat16* q;     // [N_rows, d] packed query rows
  __nv_bfloat16* out;         // [N_rows, d]
  const int* cand_off;        // device [R + 1]
  const int* kv_off;          // device [R + 1] cache row offsets
  const int* kv_len;          // device [R]
  int n_cand, S, d;
  int group;                  // query heads per K/V head
  float scale_log2;           // log2(e) / sqrt(d_h)
  int* status;
  int tiles_per_cta;          // 2 (query-tile pairs) or 1 (every tile splits its keys)
};

// Shared-memory ring and TMEM layout of enc_fa_kernel (one 128-row query tile
// per CTA, two S and two P buffers).
template <int DH>
struct FaShape {
  static constexpr int ROW_BYTES = DH * 2;                  // 64 or 128: one swizzle row
  static constexpr uint32_t SW = DH == 64 ? 2u : 4u;        // 128-byte or 64-byte swizzle
  static constexpr int ATOM = 8 * ROW_BYTES;                // 8 rows
  static constexpr int KV_BYTES = BKV * ROW_BYTES;
  static constexpr int SMEM = 2 * STG * KV_BYTES + 1024 + 256;
  // TMEM columns: S_0, S_1 (fp32, 128 each), O (fp32, DH), P_0, P_1 (bf16
  // pairs, 64 each), Q (bf16 pairs, DH / 2)
  static constexpr uint32_t T_S = 0, T_O = 256, T_P = 320, T_Q = 448;
  static constexpr int TMEM_COLS = 512;
  static_assert(T_O + DH <= T_P && T_Q + DH / 2 <= TMEM_COLS, "TMEM columns");
};

// ------------------------------------------------------------------ two query tiles per CTA

// FULL cross-attention with two 128-row query tiles (A, B) of one request and
// head per CTA.  Both tiles use each staged K/V tile, and two softmax warp
// groups (warps 2-5: tile A, warps 6-9: tile B) take turns with the tensor
// core: the MMA warp issues S_A(j), S_B(j), then, as each group hands over
// its P(j), that group's P V(j) immediately followed by its S(j+1), so one
// group computes exponentials while the other's products run.
// TMEM per tile: S (128 columns fp32; P, bf16, is written over its first 64
// columns once S has been read: the next S of the tile is issued after the P V
// that reads P, and one thread's MMAs run in issue order), O (d_h columns),
// Q (d_h / 2 columns).  A CTA whose second tile would be empty (the last of
// an odd number, often only the S context rows) splits its key range
// instead: group A takes the first ceil(nkv / 2) key tiles and group B the
// rest, both for the same query rows, and group A merges the two partial
// softmax states (O, running max, row sum) at the end through shared memory
// (a two-part form of the same online softmax).  The softmax holds a whole score row
// (128 keys) in registers after one TMEM load, takes its maximum with
// three-source max and forms the exponent arguments and row sums two lanes at
// a time (f32x2 arithmetic).  Online softmax with the stale-maximum rule
// described at the top of this file.
constexpr int PAIR_THREADS = 320;

template <int DH>
struct PairShape {
  static constexpr int ROW_BYTES = DH * 2;
  static constexpr uint32_t SW = DH == 64 ? 2u : 4u;
  static constexpr int ATOM = 8 * ROW_BYTES;
  static constexpr int KV_BYTES = BKV * ROW_BYTES;
  static constexpr int XSTRIDE = DH + 1;                   // floats per exchange row (padded)
  static constexpr int XCHG = BQ * (XSTRIDE + 2) * 4;       // O rows, running max, row sum of group B
  static constexpr int SMEM = 2 * STG * KV_BYTES + 256 + XCHG + 1024;
  static constexpr uint32_t T_S = 0, T_O = 256, T_Q = 256 + 2 * 64;
  static constexpr int TMEM_COLS = 512;
  static_assert(T_Q + 2 * (DH / 2) <= TMEM_COLS, "TMEM columns");
};

template <int DH>
__global__ void __launch_bounds__(PAIR_THREADS, 1)
    fa_pair_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV, const FaArgs a) {
  using Sh = PairShape<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sK = smem;
  uint8_t* sV = sK + STG * Sh::KV_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sV + STG * Sh::KV_BYTES);
  uint64_t* kv_full = bars;
  uint64_t* kv_empty = kv_full + STG;
  uint64_t* s_full = kv_empty + STG;     // [2] S_t(j) in TMEM (P V_t(j-1) complete too)
  uint64_t* p_full = s_full + 2;         // [2] P_t(j) written
  uint64_t* o_done = p_full + 2;         // [2] the last P V_t complete
  uint64_t* q_ready = o_done + 2;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(q_ready + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
  float* xo = reinterpret_cast<float*>(bars + 32);   // [BQ][XSTRIDE] O of group B (split keys)
  float* xm = xo + BQ * Sh::XSTRIDE;                 // [BQ] running max of group B
  float* xl = xm + BQ;                               // [BQ] row sum of group B

  pdl_launch_dependents();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qp = blockIdx.x, r = blockIdx.y, h = blockIdx.z;
  const int c0 = a.cand_off[r];
  const int M = a.cand_off[r + 1] - c0;
  const int n_q = M + a.S;
  const int tile0 = qp * a.tiles_per_cta;           // first query tile of this CTA
  if (tile0 * BQ >= n_q) return;                    // uniform: no tile here
  const int len = a.kv_len[r];
  const int kv0 = a.kv_off[r];
  const int nkv = (len + BKV - 1) / BKV;
  if (nkv <= 0) {
    if (threadIdx.x == 0) latch_status(a.status, TXS_ERR_BOUNDS);
    return;
  }
  // a lone query tile with at least two key tiles splits its keys over the
  // two groups; otherwise each group has a query tile and sees every key tile
  const bool lone = a.tiles_per_cta == 1 || (tile0 + 1) * BQ >= n_q;
  const bool split = lone && nkv >= 2;
  const int n_t = lone && !split ? 1 : 2;            // softmax groups in use (uniform)
  const int n_a = split ? (nkv + 1) / 2 : nkv;       // key tiles of group A
  // key-tile sequence of the ring: pairs, u = i (both groups read it); split
  // keys, u = 2 i + t (group t's i-th key tile; A: tile i, B: tile n_a + i)
  auto iters = [&](int t) { return split ? (t == 0 ? n_a : nkv - n_a) : nkv; };
  auto seq = [&](int t, int i) { return split ? 2 * i + t : i; };
  auto key_tile = [&](int t, int i) { return split && t == 1 ? n_a + i : i; };

  if (threadIdx.x == 0) {
    for (int st = 0; st < STG; ++st) {
      mbar_init(kv_full + st, 1);
      mbar_init(kv_empty + st, 1);
    }
    for (int t = 0; t < 2; ++t) {
      mbar_init(s_full + t, 1);
      mbar_init(p_full + t, 4);
      mbar_init(o_done + t, 1);
    }
    mbar_init(q_ready, 4 * n_t);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(tmem_holder, Sh::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;

  if (warp == 0) {
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
      int issued = 0;
      for (int j = 0; j < nkv; ++j) {
        const int st = j % STG;
        if (!mbar_wait<false>(kv_empty + st, ((j / STG) & 1) ^ 1, abort_flag)) break;
        mbar_expect_tx(kv_full + st, 2 * Sh::KV_BYTES);
        const int kt = split ? ((j & 1) ? n_a + (j >> 1) : (j >> 1)) : j;   // j-th tile of the sequence
        tma_load_2d(sK + st * Sh::KV_BYTES, &tmK, kv_full + st, (h / a.group) * DH, kv0 + kt * BKV);
        tma_load_2d(sV + st * Sh::KV_BYTES, &tmV, kv_full + st, (h / a.group) * DH, kv0 + kt * BKV);
        issued = j + 1;
      }
      if (*abort_flag)
        for (int k = issued > STG ? issued - STG : 0; k < issued; ++k)
          mbar_wait_plain<false>(kv_full + k % STG, (k / STG) & 1);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t id_s = idesc_bf16(BQ, BKV, false);
      constexpr uint32_t id_pv = idesc_bf16(BQ, DH, true);
      auto qk = [&](int t, int u) {
        const uint32_t k_addr = smem_u32(sK + (u % STG) * Sh::KV_BYTES);
#pragma unroll
        for (int k = 0; k < DH / 16; ++k) {
          const uint64_t kd = sdesc(k_addr + k * 32, 16, Sh::ATOM, Sh::SW);
          mma_bf16_ts(tmem + Sh::T_S + BKV * t, tmem + Sh::T_Q + (DH / 2) * t + 8 * k, kd, id_s, k > 0 ? 1u : 0u);
        }
        mma_commit(s_full + t);
      };
      auto pv = [&](int t, int u, bool acc) {
        const uint32_t v_addr = smem_u32(sV + (u % STG) * Sh::KV_BYTES);
#pragma unroll
        for (int k = 0; k < BKV / 16; ++k) {
          const uint64_t vd = sdesc(v_addr + k * 16 * Sh::ROW_BYTES, Sh::ATOM, Sh::ATOM, Sh::SW);
          mma_bf16_ts(tmem + Sh::T_O + 64 * t, tmem + Sh::T_S + BKV * t + 8 * k, vd, id_pv,
                      (acc || k > 0) ? 1u : 0u);
        }
      };
      bool ok = mbar_wait<false>(q_ready, 0, abort_flag);
      for (int t = 0; t < n_t && ok; ++t) {
        const int u = seq(t, 0);
        if (t == 0 || split) ok = mbar_wait<false>(kv_full + u % STG, (u / STG) & 1, abort_flag);
        if (ok) {
          tc_fence_after();
          qk(t, u);
        }
      }
      const int n_it = iters(0);               // group A has at least as many key tiles as B
      for (int i = 0; i < n_it && ok; ++i) {
        for (int t = 0; t < n_t && ok; ++t) {
          if (i >= iters(t)) continue;
          const int u = seq(t, i);
          if (!mbar_wait<false>(p_full + t, i & 1, abort_flag)) { ok = false; break; }
          tc_fence_after();
          pv(t, u, i > 0);
          // a key tile is released once every product that reads it is issued
          if (split || t == n_t - 1) mma_commit(kv_empty + u % STG);
          if (i + 1 < iters(t)) {
            const int un = seq(t, i + 1);
            if ((t == 0 || split) && !mbar_wait<false>(kv_full + un % STG, (un / STG) & 1, abort_flag)) {
              ok = false;
              break;
            }
            tc_fence_after();
            qk(t, un);
          } else {
            mma_commit(o_done + t);
          }
        }
      }
    }
  } else {
    // ---------------- softmax: warps 2-5 tile A, warps 6-9 tile B; one query row per thread
    const int t = (warp - 2) >> 2;
    if (t >= n_t) goto done;                  // no second tile in this CTA (uniform per group)
    {
    const int qw = warp & 3;                  // TMEM lane quarter
    const int m = qw * 32 + lane;
    const int j_q = (tile0 + (split ? 0 : t)) * BQ + m;   // query index within the request
    const bool valid = j_q < n_q;
    const long long grow = j_q < M ? static_cast<long long>(c0) + j_q
                                   : a.n_cand + static_cast<long long>(r) * a.S + (j_q - M);
    const uint32_t lane_off = static_cast<uint32_t>(qw * 32) << 16;
    {
      uint32_t qv[DH / 2];
      const uint4* src = reinterpret_cast<const uint4*>(a.q + (valid ? grow : 0) * a.d + h * DH);
#pragma unroll
      for (int c = 0; c < DH / 8; ++c) {
        const uint4 v = valid ? src[c] : make_uint4(0, 0, 0, 0);
        qv[4 * c] = v.x; qv[4 * c + 1] = v.y; qv[4 * c + 2] = v.z; qv[4 * c + 3] = v.w;
      }
#pragma unroll
      for (int c = 0; c < DH / 2; c += 16) tmem_st16(tmem + Sh::T_Q + (DH / 2) * t + c + lane_off, qv + c);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(q_ready);
    }
    const uint32_t t_s = tmem + Sh::T_S + BKV * t + lane_off;
    const uint32_t t_o = tmem + Sh::T_O + 64 * t + lane_off;
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    const int n_it = iters(t);
    for (int j = 0; j < n_it && ok; ++j) {
      ok = mbar_wait<false>(s_full + t, j & 1, abort_flag);
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      if (!ok) break;
      tc_fence_after();
      const int kbase = key_tile(t, j) * BKV;
      const bool ragged = kbase + BKV > len;     // uniform
      // the whole score row in registers: one TMEM load, one wait
      float sv[BKV];
      tmem_ld128(t_s, sv);
      if (ragged) {
#pragma unroll
        for (int i = 0; i < BKV; ++i)
          if (kbase + i >= len) sv[i] = -INFINITY;
      }
      float mx4[4] = {sv[0], sv[1], sv[2], sv[3]};
#pragma unroll
      for (int i = 4; i < BKV; i += 2) mx4[(i >> 1) & 3] = fmax3(mx4[(i >> 1) & 3], sv[i], sv[i + 1]);
      const float m_tile = fmax3(fmax3(mx4[0], mx4[1], mx4[2]), mx4[3], -INFINITY) * a.scale_log2;
      const bool rescale = __any_sync(0xffffffffu, m_tile > m_run + kRescaleLog2);
      float alpha = 1.f;
      if (rescale) {
        const float m_new = fmaxf(m_run, m_tile);
        alpha = ex2(m_run - m_new);                // 0 on the first tile
        m_run = m_new;
      }
      // P (bf16 pairs) over the first 64 columns of S, which is wholly in
      // registers by now; scale-and-shift and the row sum two lanes at a time.
      // Partial sums by key index mod 8, reduced as a fixed tree.  O is
      // rescaled after P is formed (the score registers are free by then);
      // P V(j) waits for p_full, which follows both.
      const float2 sc2 = make_float2(a.scale_log2, a.scale_log2);
      const float2 nm2 = make_float2(-m_run, -m_run);
      float2 ps[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) ps[i] = make_float2(0.f, 0.f);
#pragma unroll
      for (int c32 = 0; c32 < BKV; c32 += 32) {
        uint32_t pk[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const float2 x = ffma2(make_float2(sv[c32 + 2 * i], sv[c32 + 2 * i + 1]), sc2, nm2);
          const float2 p = make_float2(ex2(x.x), ex2(x.y));
          ps[i & 3] = fadd2(ps[i & 3], p);
          __nv_bfloat162 h2 = __floats2bfloat162_rn(p.x, p.y);
          pk[i] = *reinterpret_cast<uint32_t*>(&h2);
        }
        tmem_st16(t_s + c32 / 2, pk);
      }
      if (rescale) {
        if (j >= 1) {                              // O holds P V up to j - 1 (complete: S_t(j) is)
#pragma unroll
          for (int cc = 0; cc < DH; cc += 32) {
            float ov[32];
            tmem_ld32(t_o + cc, ov);
#pragma unroll
            for (int i = 0; i < 32; ++i) ov[i] *= alpha;
            tmem_st32(t_o + cc, ov);
          }
        }
        l_run *= alpha;
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full + t);
      ps[0] = fadd2(ps[0], ps[2]);
      ps[1] = fadd2(ps[1], ps[3]);
      ps[0] = fadd2(ps[0], ps[1]);
      l_run += ps[0].x + ps[0].y;
    }
    if (ok) {
      ok = mbar_wait<false>(o_done + t, 0, abort_flag);
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    }
    // split keys: group B hands its partial state (O, running max, row sum)
    // to group A, which merges the two.  Both groups reach the named barrier
    // on every path, failed waits included.
    float f_a = 1.f, f_b = 0.f;
    if (split) {
      if (t == 1) {
        if (ok) {
          tc_fence_after();
#pragma unroll
          for (int cc = 0; cc < DH; cc += 32) {
            float ov[32];
            tmem_ld32(t_o + cc, ov);
#pragma unroll
            for (int i = 0; i < 32; ++i) xo[m * Sh::XSTRIDE + cc + i] = ov[i];
          }
          xm[m] = m_run;
          xl[m] = l_run;
        } else {
          xl[m] = -1.f;                      // no partial state: group A stores nothing
        }
      }
      asm volatile("bar.sync 1, 256;" ::: "memory");
      if (t == 1) goto done;
      ok = ok && xl[m] >= 0.f;
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      if (ok) {
        const float m_b = xm[m];
        const float m_all = fmaxf(m_run, m_b);
        f_a = ex2(m_run - m_all);
        f_b = ex2(m_b - m_all);
        l_run = l_run * f_a + xl[m] * f_b;
      }
    }
    if (ok) {
      tc_fence_after();
      const float inv = 1.f / l_run;
      __nv_bfloat16* dst = a.out + grow * a.d + h * DH;
#pragma unroll
      for (int cc = 0; cc < DH; cc += 32) {
        float ov[32];
        tmem_ld32(t_o + cc, ov);
        if (split) {
#pragma unroll
          for (int i = 0; i < 32; ++i) ov[i] = ov[i] * f_a + xo[m * Sh::XSTRIDE + cc + i] * f_b;
        }
        if (valid) {
#pragma unroll
          for (int c = 0; c < 32; c += 8) {
            float tv[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) tv[i] = ov[c + i] * inv;
            Vec16<__nv_bfloat16>::store(dst + cc + c, tv);
          }
        }
      }
    }
    }
  }
done:
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, Sh::TMEM_COLS);
  }
  if (threadIdx.x == 0 && *abort_flag) latch_status(a.status, TXS_ERR_DEVICE_TIMEOUT);
}

// ------------------------------------------------------------------ encoder self-attention

// Causal self-attention of the behavior encoder (Sec. 4.1.1: causal mask and
// a relative position bias) for the new rows of each user against that
// user's cached keys/values of the same layer (App. D incremental encoding;
// a build is the case "every row is new").  One CTA per (tile of up to 128
// new rows of one user, head); the pipeline described at the top of this
// file with 4 softmax warps, two S buffers and two P buffers in TMEM (the
// exponentials of key tile j overlap the products of tile j + 1), and:
//   * key tiles of 128 positions aligned to multiples of 128 of the user's
//     own position axis (tile jj holds positions 128 jj ...), from the tile
//     of the first row's earliest visible key to the tile of the last row;
//   * the mask (key position <= row position, inside the window) and the
//     bias beta_h[min(i - j, R - 1)] (a shared-memory table, log2 units)
//     applied by the softmax warps;
//   * the running maximum raised per row (alpha = 1 for the rows that keep
//     theirs), so that a row's arithmetic depends only on its own position
//     and the keys: a tile with no visible key leaves the row untouched
//     (P = 0).  Encoding rows incrementally therefore gives the same bytes as
//     encoding them all at once.
// The K/V storage is zero-initialised when the state is created, so key rows
// of a tile that lie beyond the user's tokens are finite (P = 0 times a
// finite value).
struct EncFaArgs {
  const __nv_bfloat16* q;  // [n, d] queries of the new rows
  __nv_bfloat16* out;      // [n, d]
  const int* in_off;       // [R + 1] new rows of user r
  const int* dst0;         // [R] slot of user r's first new row
  const int* slot_off;     // [R + 1] slots of user r
  const int* tile_off;     // [R + 1] 128-row query tiles of user r
  const float* beta;       // [H][n_rel] relative bias times log2(e)
  int n_req, n_rel, window, d;
  float scale_log2;        // log2(e) / sqrt(d_h)
  int* status;
};

constexpr int kEncMaxRel = 8192;  // bias table entries staged in shared memory

template <int DH>
struct EncFaShape {
  using Sh = FaShape<DH>;
  static constexpr int BIAS_OFF = 2 * STG * Sh::KV_BYTES;
  static constexpr int SMEM = BIAS_OFF + kEncMaxRel * 4 + 1024 + 256;
};

template <int DH>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    enc_fa_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                  const EncFaArgs a) {
  using Sh = FaShape<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sK = smem;
  uint8_t* sV = sK + STG * Sh::KV_BYTES;
  float* sB = reinterpret_cast<float*>(smem + EncFaShape<DH>::BIAS_OFF);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sB + kEncMaxRel);
  uint64_t* kv_full = bars;
  uint64_t* kv_empty = kv_full + STG;
  uint64_t* s_full = kv_empty + STG;
  uint64_t* s_free = s_full + 2;
  uint64_t* p_full = s_free + 2;
  uint64_t* pv_done = p_full + 2;
  uint64_t* q_ready = pv_done + 2;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(q_ready + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  pdl_launch_dependents();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.y;
  const int r = find_segment(a.tile_off, a.n_req, blockIdx.x);
  const int t = blockIdx.x - __ldg(a.tile_off + r);
  const int row0 = __ldg(a.in_off + r) + t * BQ;
  const int nrows = min(BQ, __ldg(a.in_off + r + 1) - row0);
  const int base = __ldg(a.slot_off + r);
  const int cap = __ldg(a.slot_off + r + 1) - base;
  const int pos0 = __ldg(a.dst0 + r) - base + t * BQ;
  if (nrows <= 0) return;                            // uniform
  if (pos0 < 0 || pos0 + nrows > cap) {              // uniform
    if (threadIdx.x == 0) latch_status(a.status, TXS_ERR_BOUNDS);
    return;
  }
  const int p_last = pos0 + nrows - 1;
  const int lo = a.window > 0 ? max(0, pos0 - a.window + 1) : 0;
  const int jb = lo / BKV;
  const int nkv = p_last / BKV - jb + 1;

  for (int i = threadIdx.x; i < a.n_rel; i += NUM_THREADS)
    sB[i] = __ldg(a.beta + static_cast<long long>(h) * a.n_rel + i);
  if (threadIdx.x == 0) {
    for (int st = 0; st < STG; ++st) {
      mbar_init(kv_full + st, 1);
      mbar_init(kv_empty + st, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(s_full + b, 1);
      mbar_init(s_free + b, 4);
      mbar_init(p_full + b, 4);
      mbar_init(pv_done + b, 1);
    }
    mbar_init(q_ready, 4);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(tmem_holder, Sh::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;

  if (warp == 0) {
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
      int issued = 0;
      for (int j = 0; j < nkv; ++j) {
        const int st = j % STG;
        if (!mbar_wait<false>(kv_empty + st, ((j / STG) & 1) ^ 1, abort_flag)) break;
        mbar_expect_tx(kv_full + st, 2 * Sh::KV_BYTES);
        const int krow = base + (jb + j) * BKV;
        tma_load_2d(sK + st * Sh::KV_BYTES, &tmK, kv_full + st, h * DH, krow);
        tma_load_2d(sV + st * Sh::KV_BYTES, &tmV, kv_full + st, h * DH, krow);
        issued = j + 1;
      }
      if (*abort_flag)
        for (int k = issued > STG ? issued - STG : 0; k < issued; ++k)
          mbar_wait_plain<false>(kv_full + k % STG, (k / STG) & 1);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t id_s = idesc_bf16(BQ, BKV, false);
      constexpr uint32_t id_pv = idesc_bf16(BQ, DH, true);
      bool ok = mbar_wait<false>(q_ready, 0, abort_flag);
      tc_fence_after();
      auto pv = [&](int tt) -> bool {
        const int bt = tt & 1, st = tt % STG;
        if (!mbar_wait<false>(p_full + bt, (tt >> 1) & 1, abort_flag)) return false;
        tc_fence_after();
        const uint32_t v_addr = smem_u32(sV + st * Sh::KV_BYTES);
#pragma unroll
        for (int k = 0; k < BKV / 16; ++k) {
          const uint64_t vd = sdesc(v_addr + k * 16 * Sh::ROW_BYTES, Sh::ATOM, Sh::ATOM, Sh::SW);
          mma_bf16_ts(tmem + Sh::T_O, tmem + Sh::T_P + 64 * bt + 8 * k, vd, id_pv, (tt > 0 || k > 0) ? 1u : 0u);
        }
        mma_commit(pv_done + bt);
        mma_commit(kv_empty + st);
        return true;
      };
      for (int j = 0; j < nkv && ok; ++j) {
        const int st = j % STG, b = j & 1;
        if (!mbar_wait<false>(kv_full + st, (j / STG) & 1, abort_flag)) break;
        if (!mbar_wait<false>(s_free + b, ((j >> 1) & 1) ^ 1, abort_flag)) break;
        tc_fence_after();
        const uint32_t k_addr = smem_u32(sK + st * Sh::KV_BYTES);
#pragma unroll
        for (int k = 0; k < DH / 16; ++k) {
          const uint64_t kd = sdesc(k_addr + k * 32, 16, Sh::ATOM, Sh::SW);
          mma_bf16_ts(tmem + Sh::T_S + BKV * b, tmem + Sh::T_Q + 8 * k, kd, id_s, k > 0 ? 1u : 0u);
        }
        mma_commit(s_full + b);
        if (j >= 1) ok = pv(j - 1);
      }
      if (ok && !*abort_flag) pv(nkv - 1);
    }
  } else {
    // ---------------- softmax warps: one query row per thread
    const int qw = warp & 3;
    const int m = qw * 32 + lane;
    const bool valid = m < nrows;
    const int p = pos0 + m;                    // this row's position on the user's axis
    const uint32_t lane_off = static_cast<uint32_t>(qw * 32) << 16;
    {
      uint32_t qv[DH / 2];
      const uint4* src = reinterpret_cast<const uint4*>(a.q + static_cast<long long>(valid ? row0 + m : row0) * a.d +
                                                        h * DH);
#pragma unroll
      for (int c = 0; c < DH / 8; ++c) {
        const uint4 v = valid ? src[c] : make_uint4(0, 0, 0, 0);
        qv[4 * c] = v.x; qv[4 * c + 1] = v.y; qv[4 * c + 2] = v.z; qv[4 * c + 3] = v.w;
      }
#pragma unroll
      for (int c = 0; c < DH / 2; c += 16) tmem_st16(tmem + Sh::T_Q + c + lane_off, qv + c);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(q_ready);
    }
    const uint32_t t_o = tmem + Sh::T_O + lane_off;
    const int R1 = a.n_rel - 1;
    const float b_far = sB[R1];
    // a warp whose 32 rows are all past the tile's last new row only keeps the
    // barrier protocol: its rows' P, O and sums are never used (each O row
    // depends on its own P row only)
    const bool idle = qw * 32 >= nrows;
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    for (int j = 0; j < nkv && ok; ++j) {
      const int b = j & 1;
      ok = mbar_wait<false>(s_full + b, (j >> 1) & 1, abort_flag);
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      if (!ok) break;
      tc_fence_after();
      if (idle) {
        __syncwarp();
        if (lane == 0) mbar_arrive(s_free + b);
        if (j >= 2) {
          ok = mbar_wait<false>(pv_done + b, ((j - 2) >> 1) & 1, abort_flag);
          ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
          if (!ok) break;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(p_full + b);
        continue;
      }
      float sv[BKV];
      tmem_ld128(tmem + Sh::T_S + BKV * b + lane_off, sv);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(s_free + b);
      // logits in log2 units: scaled score + bias where visible, -inf
      // elsewhere.  Rows past the last new row follow the same rule at their
      // would-be positions (their results are discarded), which keeps the
      // warp on one path.
      const int D0 = p - (jb + j) * BKV;       // distance to the tile's first key
      const bool all_vis = D0 >= BKV - 1 && (a.window <= 0 || D0 < a.window);
      if (__all_sync(0xffffffffu, all_vis && D0 - (BKV - 1) >= R1)) {
#pragma unroll
        for (int i = 0; i < BKV; ++i) sv[i] = fmaf(sv[i], a.scale_log2, b_far);
      } else {
#pragma unroll
        for (int i = 0; i < BKV; ++i) {
          const int dist = D0 - i;
          const bool vis = dist >= 0 && (a.window <= 0 || dist < a.window);
          sv[i] = vis ? fmaf(sv[i], a.scale_log2, sB[min(dist, R1)]) : -INFINITY;
        }
      }
      float mx8[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) mx8[i] = sv[i];
#pragma unroll
      for (int i = 8; i < BKV; ++i) mx8[i & 7] = fmaxf(mx8[i & 7], sv[i]);
#pragma unroll
      for (int w = 4; w >= 1; w >>= 1)
#pragma unroll
        for (int i = 0; i < w; ++i) mx8[i] = fmaxf(mx8[i], mx8[i + w]);
      const float m_tile = mx8[0];
      const bool need = m_tile > m_run + kRescaleLog2;
      if (__any_sync(0xffffffffu, need)) {
        const float m_new = need ? fmaxf(m_run, m_tile) : m_run;
        const float alpha = need ? ex2(m_run - m_new) : 1.f;   // 0 on a row's first visible tile
        if (j >= 1) {
          ok = mbar_wait<false>(pv_done + ((j - 1) & 1), ((j - 1) >> 1) & 1, abort_flag);
          ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
          if (!ok) break;
          tc_fence_after();
#pragma unroll
          for (int cc = 0; cc < DH; cc += 32) {
            float ov[32];
            tmem_ld32(t_o + cc, ov);
#pragma unroll
            for (int i = 0; i < 32; ++i) ov[i] *= alpha;
            tmem_st32(t_o + cc, ov);
          }
        }
        l_run *= alpha;
        m_run = m_new;
      }
      if (j >= 2) {
        ok = mbar_wait<false>(pv_done + b, ((j - 2) >> 1) & 1, abort_flag);
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        if (!ok) break;
        tc_fence_after();
      }
      // P = 2^(s - m_run); 0 where masked (also while the row has no visible key yet)
      const uint32_t t_p = tmem + Sh::T_P + 64 * b + lane_off;
      float ps8[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) ps8[i] = 0.f;
#pragma unroll
      for (int c32 = 0; c32 < BKV; c32 += 32) {
        uint32_t pk[16];
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          const float s0 = sv[c32 + i], s1 = sv[c32 + i + 1];
          const float p0 = s0 == -INFINITY ? 0.f : ex2(s0 - m_run);
          const float p1 = s1 == -INFINITY ? 0.f : ex2(s1 - m_run);
          ps8[i & 7] += p0;
          ps8[(i + 1) & 7] += p1;
          __nv_bfloat162 h2 = __floats2bfloat162_rn(p0, p1);
          pk[i / 2] = *reinterpret_cast<uint32_t*>(&h2);
        }
        tmem_st16(t_p + c32 / 2, pk);
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full + b);
#pragma unroll
      for (int w = 4; w >= 1; w >>= 1)
#pragma unroll
        for (int i = 0; i < w; ++i) ps8[i] += ps8[i + w];
      l_run += ps8[0];
    }
    if (ok) {
      ok = mbar_wait<false>(pv_done + ((nkv - 1) & 1), ((nkv - 1) >> 1) & 1, abort_flag);
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    }
    if (ok && !idle) {
      tc_fence_after();
      const float inv = valid ? 1.f / l_run : 0.f;
      __nv_bfloat16* dst = a.out + static_cast<long long>(valid ? row0 + m : row0) * a.d + h * DH;
#pragma unroll
      for (int cc = 0; cc < DH; cc += 32) {
        float ov[32];
        tmem_ld32(t_o + cc, ov);
        if (valid) {
#pragma unroll
          for (int c = 0; c < 32; c += 8) {
            float tv[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) tv[i] = ov[c + i] * inv;
            Vec16<__nv_bfloat16>::store(dst + cc + c, tv);
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, Sh::TMEM_COLS);
  }
  if (threadIdx.x == 0 && *abort_flag) latch_status(a.status, TXS_ERR_DEVICE_TIMEOUT);
}

// ------------------------------------------------------------------ host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// K or V of one layer: [rows, d] bf16, box {DH columns, 128 rows}.
template <int DH>
static bool make_kv_map(CUtensorMap* tm, const void* base, long long rows, int d) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(d) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(DH), static_cast<cuuint32_t>(BKV)};
  cuuint32_t estr[2] = {1, 1};
  return fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, DH == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int DH>
static cudaError_t launch_pair_dh(const FaArgs& a, const void* Kc, const void* Vc, long long cap_total, int n_req,
                                  int max_q_pairs, int H, int dkv, cudaStream_t s) {
  using Sh = PairShape<DH>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(fa_pair_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, Sh::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  CUtensorMap tk, tv;
  if (!make_kv_map<DH>(&tk, Kc, cap_total, dkv) || !make_kv_map<DH>(&tv, Vc, cap_total, dkv))
    return cudaErrorInvalidValue;
  return launch_pdl(fa_pair_kernel<DH>, dim3(max_q_pairs, n_req, H), dim3(PAIR_THREADS), Sh::SMEM, s, tk, tv, a);
}

template <int DH>
static cudaError_t launch_enc_dh(const EncFaArgs& a, const void* K, const void* V, long long cap_total, int n_tiles,
                                 int H, cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(enc_fa_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         EncFaShape<DH>::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  CUtensorMap tk, tv;
  if (!make_kv_map<DH>(&tk, K, cap_total, a.d) || !make_kv_map<DH>(&tv, V, cap_total, a.d))
    return cudaErrorInvalidValue;
  return launch_pdl(enc_fa_kernel<DH>, dim3(n_tiles, H), dim3(NUM_THREADS), EncFaShape<DH>::SMEM, s, tk, tv, a);
}

}  // namespace fa

bool enc_attn_tc_supported(int d, int H, int n_rel) {
  const int dh = d / H;
  return (dh == 32 || dh == 64) && n_rel >= 1 && n_rel <= fa::kEncMaxRel && d % 8 == 0;
}

cudaError_t launch_enc_attn_tc(const __nv_bfloat16* q, const __nv_bfloat16* K, const __nv_bfloat16* V,
                               __nv_bfloat16* out, long long cap_total, const int* in_off, const int* dst0,
                               const int* slot_off, const int* tile_off, int n_req, int n_tiles,
                               const float* beta_log2, int n_rel, int window, int H, int d, int* status,
                               cudaStream_t s) {
  if (n_tiles == 0) return cudaSuccess;
  if (!enc_attn_tc_supported(d, H, n_rel)) return cudaErrorNotSupported;
  const int dh = d / H;
  fa::EncFaArgs a{q, out, in_off, dst0, slot_off, tile_off, beta_log2, n_req, n_rel, window, d,
                  1.4426950408889634f / sqrtf(static_cast<float>(dh)), status};
  prof_begin(KC_ENC_ATTN, s);
  cudaError_t err = dh == 64 ? fa::launch_enc_dh<64>(a, K, V, cap_total, n_tiles, H, s)
                             : fa::launch_enc_dh<32>(a, K, V, cap_total, n_tiles, H, s);
  prof_end(KC_ENC_ATTN, s);
  return err;
}

bool fa_full_supported(int d, int H, long long cap_total) {
  const int dh = d / H;
  return (dh == 32 || dh == 64) && cap_total >= fa::BKV && d % 8 == 0;
}

cudaError_t launch_fa_full(const __nv_bfloat16* q, __nv_bfloat16* out, const __nv_bfloat16* Kc,
                           const __nv_bfloat16* Vc, long long cap_total, const int* cand_off_dev,
                           const int* cand_off_host, const int* kv_off, const int* kv_len, int n_req, int n_cand,
                           int S, int H, int Hkv, int d, int* status, cudaStream_t s) {
  int max_q = 0;
  for (int r = 0; r < n_req; ++r) max_q = std::max(max_q, cand_off_host[r + 1] - cand_off_host[r] + S);
  if (max_q == 0) return cudaSuccess;
  if (Hkv < 1 || H % Hkv) return cudaErrorInvalidValue;
  const int dh = d / H;
  fa::FaArgs a{q, out, cand_off_dev, kv_off, kv_len, n_cand, S, d, H / Hkv,
               1.4426950408889634f / sqrtf(static_cast<float>(dh)), status, 2};
  const int tiles = (max_q + fa::BQ - 1) / fa::BQ;
  prof_begin(KC_ATTN_CROSS, s);
  cudaError_t err;
  // two query tiles per CTA share each K/V tile when the pairs still fill
  // the GPU; otherwise (few requests: a single request would leave most SMs
  // idle) one query tile per CTA, its key tiles split over the two groups
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
      sms = 152;
  }
  const long long pair_ctas = static_cast<long long>((tiles + 1) / 2) * n_req * H;
  a.tiles_per_cta = tiles >= 2 && pair_ctas >= 2LL * sms ? 2 : 1;
  const int grid_x = (tiles + a.tiles_per_cta - 1) / a.tiles_per_cta;
  err = dh == 64 ? fa::launch_pair_dh<64>(a, Kc, Vc, cap_total, n_req, grid_x, H, Hkv * dh, s)
                 : fa::launch_pair_dh<32>(a, Kc, Vc, cap_total, n_req, grid_x, H, Hkv * dh, s);
  prof_end(KC_ATTN_CROSS, s);
  return err;
}

}  // namespace txs
