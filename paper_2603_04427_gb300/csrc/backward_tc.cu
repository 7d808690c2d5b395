// Gradient kernel of thin-key attention on the 5th-generation tensor cores
// (r <= 64): tcgen05.mma with accumulators in tensor memory, operands staged
// in shared memory by TMA.
//
// Paper: Section 2.1, Eqs. 1-4 (the forward being differentiated); training
// with thin keys is Sections 3.2-3.3.  Per head, with p = softmax(scale q k^T)
// (masked) and dL/d(out) = dO:
//     dV = p^T dO,  dP = dO v^T,  dS = p * (dP - D),  D_i = sum_c dO_ic out_ic,
//     dQ = scale dS k,  dK = scale dS^T q.
// The preprocessing pass (backward.cu) has written D and lse2 = lse log2(e)
// for every query row, padded to a multiple of 128 rows (lse2 = +inf, D = 0 on
// the padding), and zeroed dQ.
//
// One CTA per (sequence, kv head g, 128-key tile j).  Keys are the MMA's M
// dimension and the TMEM lanes: thread t of a 4-warp group owns key t.  The
// CTA visits every 128-query tile i (i >= j when causal) of each of the G
// query heads of g, as two 64-query halves h:
//   warp 12 (one lane): TMA loads of K_j, V_j (once) and, per tile, of Q_i,
//       dO_i and the rows' lse2 / D into a 2-stage ring.
//   warp 13 (whole warp, one elected lane issues): per tile and half
//       S^T_h  = K Q_h^T     (M=128 keys, N=64 queries, K=r)
//       dP^T_h = V dO_h^T    (M=128, N=64, K=d_v)
//       dV    += P^T_h dO_h  (N=d_v, K=64; P^T_h read from TMEM)
//       dK    += dS^T_h Q_h  (N=r,   K=64; dS^T_h from shared memory, K-major)
//     and per tile  dQ_i = dS K  (M=128 queries, N=r, K=128 keys; dS from the
//     same shared-memory tile read MN-major), completion on mbarriers through
//     tcgen05.commit.  The next tile's S / dP products of a half are issued as
//     soon as that half's P has been consumed, so one half's softmax overlaps
//     the other half's products.
//   warps 0-3 / 4-7 (half 0 / 1): read S^T_h and dP^T_h from TMEM, form
//       P^T = exp2(S^T scale log2e - lse2) (masked) and dS^T = P^T (dP^T - D),
//       write P^T as bf16 into TMEM over S^T_h and dS^T as bf16 into the
//       swizzled shared-memory tile.
//   warps 8-11 (thread t owns query t of the tile): read dQ_i from TMEM and
//       add it into global dq with one bulk reduce-add per row
//       (cp.reduce.async.bulk .add.f32); at the end, dK (times scale) and dV
//       of the CTA's keys from TMEM to global memory.
//
// TMEM columns: [0,64) S^T_0 (P^T_0 in its first 32), [64,128) dP^T_0,
// [128,192) S^T_1, [192,256) dP^T_1, then dV (d_v), dK (r), dQ (r).
#include <algorithm>
#include <type_traits>

#include "common.cuh"
#include "kernels.h"
#include "tc05.cuh"

namespace tk {
namespace {

constexpr int kKeys = 128;         // keys per CTA (MMA M, TMEM lanes)
constexpr int kQT = 128;           // queries per tile
constexpr int kHalfQ = 64;         // queries per S / dP half
constexpr int kTcThreads = 448;    // 3 x 4 warps, the TMA warp, the MMA warp
constexpr int kTmemColsTc = 512;
constexpr int kBoxB = 128 * 128;   // one 64-column (128-byte) box of a 128-row tile

constexpr int align1k(int x) { return (x + 1023) / 1024 * 1024; }

template <int R, int DV>
struct TCfg {
  static_assert(R <= 64, "thin keys only: the r = 128 backward runs on mma.sync");
  // Q / K rows are r bf16 = 2r bytes, one swizzle span (32, 64 or 128 bytes)
  static constexpr int QK_SW = 2 * R;
  static constexpr uint32_t QK_LAYOUT = QK_SW == 32 ? 6u : (QK_SW == 64 ? 4u : 2u);
  static constexpr int KB = kKeys * R * 2;         // K tile
  static constexpr int VB = kKeys * DV * 2;        // V tile (DV / 64 boxes)
  static constexpr int QB = kQT * R * 2;           // Q tile
  static constexpr int OB = kQT * DV * 2;          // dO tile (DV / 64 boxes)
  static constexpr int ST_Q = 0, ST_O = align1k(QB), ST_LSE = ST_O + OB, ST_D = ST_LSE + kQT * 4;
  static constexpr int STAGE = ST_D + kQT * 4;      // multiple of 1024
  static constexpr int DSB = kKeys * kQT * 2;      // dS^T tile: [2 halves][128 keys][64 queries]
  // dQ rows staged for the bulk reduce, rows padded by 16 bytes so that the
  // rows' 16-byte stores of one instruction fall in different banks
  static constexpr int DQ_ROW = R * 4 + 16;
  static constexpr int DQB = kQT * DQ_ROW;
  static constexpr int OFF_K = 0;
  static constexpr int OFF_V = align1k(KB);
  static constexpr int OFF_ST = OFF_V + VB;
  static constexpr int OFF_DS = OFF_ST + 2 * STAGE;
  static constexpr int BASE = OFF_DS + DQB + 256 + 1024;  // without dS tiles; + barriers, alignment slack
  static constexpr int NDS = BASE + 2 * DSB <= 227 * 1024 ? 2 : 1;  // dS^T tiles in flight
  static constexpr int OFF_DQ = OFF_DS + NDS * DSB;
  static constexpr int OFF_BAR = OFF_DQ + DQB;
  // at least 116 KB so that one CTA (and its 512 TMEM columns) sits on an SM alone
  static constexpr int SMEM = std::max(OFF_BAR + 256 + 1024, 116 * 1024);
  static_assert(OFF_BAR + 256 + 1024 <= 227 * 1024, "shared memory");
  // TMEM columns
  static constexpr int T_S = 0;          // + 128 h: S^T_h (P^T_h packed in its first 32)
  static constexpr int T_DP = 64;        // + 128 h: dP^T_h
  static constexpr int T_DV = 256, T_DK = 256 + DV, T_DQ = 256 + DV + R;
  static_assert(T_DQ + R <= kTmemColsTc, "TMEM columns");
  // instruction descriptors
  static constexpr uint32_t ID_S = instr_desc(kKeys, kHalfQ, false);       // S^T, dP^T
  static constexpr uint32_t ID_DV = instr_desc(kKeys, DV, true);           // A = P^T (TMEM), B = dO MN-major
  static constexpr uint32_t ID_DK = instr_desc(kKeys, R, true);            // A = dS^T K-major, B = Q MN-major
  static constexpr uint32_t ID_DQ = instr_desc(kQT, R, true, true);        // A = dS MN-major, B = K MN-major
};

struct TcMaps {
  CUtensorMap q, k, v, d_out;
};

__device__ __forceinline__ void bulk_reduce_add_f32(float* gdst, const void* ssrc, uint32_t bytes) {
  asm volatile("cp.reduce.async.bulk.global.shared::cta.bulk_group.add.f32 [%0], [%1], %2;" ::"l"(gdst),
               "r"(smem_addr(ssrc)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_all() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// 32 consecutive columns at each of two TMEM addresses, one wait.
__device__ __forceinline__ void tmem_ld32x2(uint32_t ta, uint32_t tb, uint32_t* v) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, "
      "%28, %29, %30, %31}, [%64];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%32, %33, %34, %35, %36, %37, %38, %39, %40, "
      "%41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, "
      "%58, %59, %60, %61, %62, %63}, [%65];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : TK_R8(0), TK_R8(8), TK_R8(16), TK_R8(24), TK_R8(32), TK_R8(40), TK_R8(48), TK_R8(56)
      : "r"(ta), "r"(tb)
      : "memory");
}
// N consecutive 32-bit columns (N = 16, 32 or 64).
template <int N>
__device__ __forceinline__ void tmem_ld_n(uint32_t taddr, uint32_t* v) {
  if constexpr (N == 16) tmem_ld16(taddr, v);
  else if constexpr (N == 32) tmem_ld32(taddr, v);
  else tmem_ld64(taddr, v);
}

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);  // low half = lo
  return *reinterpret_cast<uint32_t*>(&v);
}

template <int R, int DV>
__global__ void __launch_bounds__(kTcThreads, 1)
bwd_tc_kernel(const __grid_constant__ TcMaps maps, const BackwardParams p) {
  using C = TCfg<R, DV>;
  constexpr int NDS = C::NDS;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* kv_full = bars + 0;
  uint64_t* qd_full = bars + 1;      // [2] stage loaded
  uint64_t* qd_empty = bars + 3;     // [2] stage consumed
  uint64_t* s_full = bars + 5;       // [2] S^T_h, dP^T_h in TMEM
  uint64_t* p_ready = bars + 7;      // [2] P^T_h in TMEM, dS^T_h in shared memory
  uint64_t* ds_free = bars + 9;      // [NDS] dS^T tile read by its last product
  uint64_t* dq_full = bars + 11;
  uint64_t* dq_empty = bars + 12;
  uint64_t* acc_full = bars + 13;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 14);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int S = p.S, G = p.Hq / p.Hkv;
  const int n_kt = (S + kKeys - 1) / kKeys;
  const int n_qt = (S + kQT - 1) / kQT;
  // CTA order: (sequence, kv head) major, the key tiles with most work first
  const int j = static_cast<int>(blockIdx.x % n_kt);
  const int bg = static_cast<int>(blockIdx.x / n_kt);
  const int b = bg / p.Hkv, g = bg % p.Hkv;
  const int i0 = p.causal ? j : 0;     // kKeys == kQT: query tiles i >= j see key tile j
  const int per_head = n_qt - i0;
  const int n_tiles = G * per_head;
  auto tile_head = [&](int t) { return g * G + t / per_head; };
  auto tile_q = [&](int t) { return i0 + t % per_head; };

  if (tid == 0) {
    mbar_init(kv_full, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(&qd_full[s], 1);
      mbar_init(&qd_empty[s], 1);
      mbar_init(&s_full[s], 1);
      mbar_init(&p_ready[s], 128);
    }
    for (int s = 0; s < NDS; ++s) mbar_init(&ds_free[s], 1);
    mbar_init(dq_full, 1);
    mbar_init(dq_empty, 128);
    mbar_init(acc_full, 1);
    fence_barrier_init();
  }
  if (warp == 13) {
    tmem_alloc(tmem_slot, kTmemColsTc);
    tmem_relinquish();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 12) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0) {
      const int kv_plane = b * p.Hkv + g;
      prefetch_map(&maps.q);
      prefetch_map(&maps.k);
      prefetch_map(&maps.v);
      prefetch_map(&maps.d_out);
      mbar_arrive_expect_tx(kv_full, C::KB + C::VB);
      tma_load_3d(smem + C::OFF_K, &maps.k, 0, j * kKeys, kv_plane, kv_full);
      for (int x = 0; x < DV / 64; ++x)
        tma_load_3d(smem + C::OFF_V + x * kBoxB, &maps.v, 64 * x, j * kKeys, kv_plane, kv_full);
      int issued = 0;
      for (int t = 0; t < n_tiles; ++t) {
        const int st = t & 1;
        if (t >= 2 && !mbar_wait(&qd_empty[st], ((t >> 1) - 1) & 1, p.err)) break;
        const int bh = b * p.Hq + tile_head(t), i = tile_q(t);
        unsigned char* sb = smem + C::OFF_ST + st * C::STAGE;
        mbar_arrive_expect_tx(&qd_full[st], C::QB + C::OB + 2 * kQT * 4);
        tma_load_3d(sb + C::ST_Q, &maps.q, 0, i * kQT, bh, &qd_full[st]);
        for (int x = 0; x < DV / 64; ++x)
          tma_load_3d(sb + C::ST_O + x * kBoxB, &maps.d_out, 64 * x, i * kQT, bh, &qd_full[st]);
        const size_t srow = static_cast<size_t>(bh) * p.S_pad + static_cast<size_t>(i) * kQT;
        bulk_g2s(sb + C::ST_LSE, p.lse2 + srow, kQT * 4, &qd_full[st]);
        bulk_g2s(sb + C::ST_D, p.dsum + srow, kQT * 4, &qd_full[st]);
        issued = t + 1;
      }
      // no copy may still be landing in shared memory when the CTA exits
      // (normally all were consumed; after a timed-out wait, bounded waits)
      mbar_wait(kv_full, 0, p.err);
      for (int t = std::max(0, issued - 2); t < issued; ++t) mbar_wait(&qd_full[t & 1], (t >> 1) & 1, p.err);
    }
  } else if (warp == 13) {
    // ------------------------------------------------------------------ MMA issuer
    const uint32_t s_base = smem_addr(smem);
    // one descriptor serves a tile read K-major and MN-major: SBO is the stride of
    // 8-row groups either way, LBO the stride of MN atoms (unused when N fits one)
    const Desc dK_d = make_desc(s_base + C::OFF_K, 16, 8 * C::QK_SW, C::QK_LAYOUT);     // K
    const Desc dV_a = make_desc(s_base + C::OFF_V, 16, 1024, 2u);                       // V, K-major
    const Desc dQ_b = make_desc(s_base + C::OFF_ST + C::ST_Q, 16, 8 * C::QK_SW, C::QK_LAYOUT);     // Q
    const Desc dO_bk = make_desc(s_base + C::OFF_ST + C::ST_O, 16, 1024, 2u);           // dO, K-major
    const Desc dO_bm = make_desc(s_base + C::OFF_ST + C::ST_O, kBoxB, 1024, 2u);        // dO, MN-major
    const Desc dS_ak = make_desc(s_base + C::OFF_DS, 16, 1024, 2u);                     // dS^T, K-major
    const Desc dS_am = make_desc(s_base + C::OFF_DS, C::DSB / 2, 1024, 2u);             // dS, MN-major
    auto issue_sdp = [&](int t, int h) {   // S^T_h, dP^T_h of tile t
      const uint32_t so = (t & 1) * C::STAGE;
#pragma unroll
      for (int k = 0; k < R / 16; ++k)
        mma_ss_e(tmem + C::T_S + 128 * h, dK_d.at(k * 32), dQ_b.at(so + h * kHalfQ * C::QK_SW + k * 32),
                 C::ID_S, k > 0);
#pragma unroll
      for (int k = 0; k < DV / 16; ++k) {
        const uint32_t ko = (k / 4) * kBoxB + (k % 4) * 32;
        mma_ss_e(tmem + C::T_DP + 128 * h, dV_a.at(ko), dO_bk.at(so + ko + h * kHalfQ * 128), C::ID_S, k > 0);
      }
      tc_commit_e(&s_full[h]);
    };
    auto issue_dvdk = [&](int t, int h) {  // dV += P^T_h dO_h, dK += dS^T_h Q_h
      const uint32_t so = (t & 1) * C::STAGE;
      const uint32_t dso = (t % NDS) * C::DSB + h * (C::DSB / 2);
#pragma unroll
      for (int kk = 0; kk < kHalfQ / 16; ++kk)
        mma_ts_e(tmem + C::T_DV, tmem + C::T_S + 128 * h + 8 * kk,
                 dO_bm.at(so + (h * kHalfQ + 16 * kk) * 128), C::ID_DV, (t > 0 || h > 0 || kk > 0) ? 1u : 0u);
#pragma unroll
      for (int kk = 0; kk < kHalfQ / 16; ++kk)
        mma_ss_e(tmem + C::T_DK, dS_ak.at(dso + kk * 32),
                 dQ_b.at(so + (h * kHalfQ + 16 * kk) * C::QK_SW), C::ID_DK, (t > 0 || h > 0 || kk > 0) ? 1u : 0u);
    };
    bool ok = __all_sync(0xffffffffu, mbar_wait(kv_full, 0, p.err) && mbar_wait(&qd_full[0], 0, p.err));
    if (ok) {
      tc_fence_after();
      issue_sdp(0, 0);
      issue_sdp(0, 1);
    }
    for (int t = 0; ok && t < n_tiles; ++t) {
      const bool next = t + 1 < n_tiles;
      if (!(ok = __all_sync(0xffffffffu, mbar_wait(&p_ready[0], t & 1, p.err)))) break;
      tc_fence_after();
      issue_dvdk(t, 0);
      if (next) {
        if (!(ok = __all_sync(0xffffffffu, mbar_wait(&qd_full[(t + 1) & 1], ((t + 1) >> 1) & 1, p.err)))) break;
        tc_fence_after();
        issue_sdp(t + 1, 0);
      }
      if (!(ok = __all_sync(0xffffffffu, mbar_wait(&p_ready[1], t & 1, p.err)))) break;
      tc_fence_after();
      issue_dvdk(t, 1);
      if (t > 0 && !(ok = __all_sync(0xffffffffu, mbar_wait(dq_empty, (t - 1) & 1, p.err)))) break;
      tc_fence_after();
      {  // dQ_t = dS K over the 128 keys
        const uint32_t dso = (t % NDS) * C::DSB;
#pragma unroll
        for (int k = 0; k < kKeys / 16; ++k)
          mma_ss_e(tmem + C::T_DQ, dS_am.at(dso + k * 16 * 128), dK_d.at(k * 16 * C::QK_SW), C::ID_DQ, k > 0);
      }
      tc_commit_e(dq_full);
      tc_commit_e(&ds_free[t % NDS]);
      tc_commit_e(&qd_empty[t & 1]);
      if (next) issue_sdp(t + 1, 1);
    }
    if (ok) tc_commit_e(acc_full);
  } else if (warp < 8) {
    // ------------------------------------------------------------------ softmax gradient warps
    const int h = warp >> 2;                      // query half
    const int kt = (warp & 3) * 32 + lane;        // key of this thread within the tile (TMEM lane)
    const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t tS = tmem + C::T_S + 128 * h + lane_off, tD = tmem + C::T_DP + 128 * h + lane_off;
    const bool kvalid = j * kKeys + kt < S;
    const float sl2 = p.scale * 1.4426950408889634f;
    for (int t = 0; t < n_tiles; ++t) {
      const int st = t & 1, buf = t % NDS;
      bool ok = mbar_wait(&s_full[h], t & 1, p.err) && mbar_wait(&qd_full[st], (t >> 1) & 1, p.err);
      if (ok && t >= NDS) ok = mbar_wait(&ds_free[buf], ((t / NDS) - 1) & 1, p.err);
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      const unsigned char* sb = smem + C::OFF_ST + st * C::STAGE;
      const float* lse2 = reinterpret_cast<const float*>(sb + C::ST_LSE) + h * kHalfQ;
      const float* dsum = reinterpret_cast<const float*>(sb + C::ST_D) + h * kHalfQ;
      unsigned char* ds_row = smem + C::OFF_DS + buf * C::DSB + h * (C::DSB / 2) + kt * 128;
      // keys past S, and keys after the query on the diagonal tile, get weight 0
      const int qlim = (p.causal && tile_q(t) == j) ? kt - h * kHalfQ : 0;  // visible iff column >= qlim
      // warp-uniform choice: both paths issue warp-collective TMEM loads and stores
      const bool masked = __any_sync(0xffffffffu, !kvalid || qlim > 0);
      auto chunk = [&](auto mask_tag, int c) {
        constexpr bool kMask = decltype(mask_tag)::value;
        uint32_t v[64];   // [0, 32): S^T, [32, 64): dP^T
        tmem_ld32x2(tS + 32 * c, tD + 32 * c, v);
        uint32_t pk[16], dk[16];
#pragma unroll
        for (int e2 = 0; e2 < 16; ++e2) {
          float pr[2], dsv[2];
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const int e = 2 * e2 + u, col = 32 * c + e;
            float x = __uint_as_float(v[e]) * sl2 - lse2[col];
            if (kMask && (!kvalid || col < qlim)) x = -INFINITY;
            pr[u] = fast_exp2(x);
            dsv[u] = pr[u] * (__uint_as_float(v[32 + e]) - dsum[col]);
          }
          pk[e2] = pack2(pr[0], pr[1]);
          dk[e2] = pack2(dsv[0], dsv[1]);
        }
        tmem_st16(tS + 16 * c, pk);
        // dS^T row kt, queries 32c .. 32c+31 of the half: four 16-byte chunks, SW128 swizzle
#pragma unroll
        for (int m = 0; m < 4; ++m) {
          const int chunk_i = (4 * c + m) ^ (kt & 7);
          *reinterpret_cast<uint4*>(ds_row + chunk_i * 16) =
              make_uint4(dk[4 * m], dk[4 * m + 1], dk[4 * m + 2], dk[4 * m + 3]);
        }
      };
#pragma unroll
      for (int c = 0; c < kHalfQ / 32; ++c) {
        if (masked) chunk(std::true_type{}, c);
        else chunk(std::false_type{}, c);
      }
      tmem_wait_st();
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(&p_ready[h]);
    }
  } else {
    // ------------------------------------------------------------------ dQ / dK / dV epilogue
    const int row = (warp & 3) * 32 + lane;       // TMEM lane: a query (dQ) or a key (dK, dV)
    const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
    float* stage = reinterpret_cast<float*>(smem + C::OFF_DQ + row * C::DQ_ROW);
    bool ok = true;
    bool pending = false;
    for (int t = 0; t < n_tiles; ++t) {
      ok = mbar_wait(dq_full, t & 1, p.err);
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      tc_fence_after();
      uint32_t v[R];
      tmem_ld_n<R>(tmem + C::T_DQ + lane_off, v);
      tc_fence_before();
      mbar_arrive(dq_empty);
      const int i = tile_q(t);
      const int q = i * kQT + row;
      if (q < S) {
        if (pending) bulk_wait_read_all();   // the previous row's reduce has read the stage
#pragma unroll
        for (int c = 0; c < R / 4; ++c)
          reinterpret_cast<float4*>(stage)[c] =
              make_float4(__uint_as_float(v[4 * c]) * p.scale, __uint_as_float(v[4 * c + 1]) * p.scale,
                          __uint_as_float(v[4 * c + 2]) * p.scale, __uint_as_float(v[4 * c + 3]) * p.scale);
        fence_proxy_async_smem();
        const size_t x = (static_cast<size_t>(b) * p.Hq + tile_head(t)) * S + q;
        bulk_reduce_add_f32(p.dq + x * R, stage, R * 4);
        bulk_commit();
        pending = true;
      }
    }
    if (pending) bulk_wait_all();
    if (ok) ok = mbar_wait(acc_full, 0, p.err);
    if (__all_sync(0xffffffffu, ok)) {
      tc_fence_after();
      const int key = j * kKeys + row;
      const size_t kx = (static_cast<size_t>(b) * p.Hkv + g) * S + key;
      {
        uint32_t v[R];
        tmem_ld_n<R>(tmem + C::T_DK + lane_off, v);
        if (key < S) {
          float4* dst = reinterpret_cast<float4*>(p.dk + kx * R);
#pragma unroll
          for (int c = 0; c < R / 4; ++c)
            dst[c] = make_float4(__uint_as_float(v[4 * c]) * p.scale, __uint_as_float(v[4 * c + 1]) * p.scale,
                                 __uint_as_float(v[4 * c + 2]) * p.scale, __uint_as_float(v[4 * c + 3]) * p.scale);
        }
      }
#pragma unroll
      for (int c0 = 0; c0 < DV / 32; ++c0) {
        uint32_t v[32];
        tmem_ld32(tmem + C::T_DV + lane_off + 32 * c0, v);
        if (key < S) {
          float4* dst = reinterpret_cast<float4*>(p.dv + kx * DV + 32 * c0);
#pragma unroll
          for (int c = 0; c < 8; ++c)
            dst[c] = make_float4(__uint_as_float(v[4 * c]), __uint_as_float(v[4 * c + 1]),
                                 __uint_as_float(v[4 * c + 2]), __uint_as_float(v[4 * c + 3]));
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 13) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemColsTc);
  }
}

template <int R, int DV>
cudaError_t launch_tc(const BackwardParams& p, cudaStream_t stream) {
  using C = TCfg<R, DV>;
  TcMaps maps;
  if (!make_map(&maps.q, p.q, R, p.S, p.B * p.Hq, R, kQT, C::QK_SW) ||
      !make_map(&maps.k, p.k, R, p.S, p.B * p.Hkv, R, kKeys, C::QK_SW) ||
      !make_map(&maps.v, p.v, DV, p.S, p.B * p.Hkv, 64, kKeys, 128) ||
      !make_map(&maps.d_out, p.d_out, DV, p.S, p.B * p.Hq, 64, kQT, 128))
    return cudaErrorInvalidValue;
  auto kern = bwd_tc_kernel<R, DV>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  const long long n_kt = (p.S + kKeys - 1) / kKeys;
  const long long grid = static_cast<long long>(p.B) * p.Hkv * n_kt;
  if (grid > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  kern<<<static_cast<unsigned>(grid), kTcThreads, C::SMEM, stream>>>(maps, p);
  return cudaGetLastError();
}

template <int R>
cudaError_t tc_by_dv(const BackwardParams& p, cudaStream_t s, int* uns) {
  switch (p.DV) {
    case 64: return launch_tc<R, 64>(p, s);
    case 128: return launch_tc<R, 128>(p, s);
  }
  *uns = 1;
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_backward_tc(const BackwardParams& p, cudaStream_t stream, int* unsupported) {
  switch (p.R) {
    case 16: return tc_by_dv<16>(p, stream, unsupported);
    case 32: return tc_by_dv<32>(p, stream, unsupported);
    case 64: return tc_by_dv<64>(p, stream, unsupported);
  }
  *unsupported = 1;
  return cudaSuccess;
}

}  // namespace tk
