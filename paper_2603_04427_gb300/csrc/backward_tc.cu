// Gradient kernel of thin-key attention on the 5th-generation tensor cores:
// tcgen05.mma with accumulators in tensor memory, operands staged in shared
// memory by TMA.
//
// Paper: Section 2.1, Eqs. 1-4 (the forward being differentiated); training
// with thin keys is Sections 3.2-3.3.  Per head, with p = softmax(scale q k^T)
// (masked) and dL/d(out) = dO:
//     dV = p^T dO,  dP = dO v^T,  dS = p * (dP - D),  D_i = sum_c dO_ic out_ic,
//     dQ = scale dS k,  dK = scale dS^T q.
// The preprocessing pass (backward.cu) has written -lse log2(e) and -D for
// every query row, padded to a multiple of 128 rows (-inf and 0 on the
// padding: such rows get weight 0), and zeroed dQ.
//
// One CTA per (sequence, kv head g, 128-key tile j).  Keys are the MMA's M
// dimension and the TMEM lanes: thread t of a 4-warp group owns key t.  The
// CTA visits every 128-query tile i (i >= j when causal) of each of the G
// query heads of g, as two 64-query halves h:
//   warp 9 (one lane): TMA loads of K_j, V_j (once) and, per half tile, of
//       Q, dO and the rows' statistics into a 4-slot ring.
//   warp 8 (whole warp, one elected lane issues): per tile and half
//       S^T_h  = K Q_h^T     (M=128 keys, N=64 queries, K=r)
//       dP^T_h = V dO_h^T    (M=128, N=64, K=d_v)
//       dV    += P^T_h dO_h  (N=d_v, K=64; P^T_h read from TMEM)
//       dK    += dS^T_h Q_h  (N=r,   K=64; dS^T_h from shared memory, K-major)
//     and per tile  dQ_i = dS K  (M=128 queries, N=r, K=128 keys; dS from the
//     same shared-memory tile read MN-major), completion on mbarriers through
//     tcgen05.commit.  Where TMEM has room for P^T in columns of its own and
//     shared memory for two dS tiles (the EARLY schedule), the next tile's
//     S / dP products of a half are issued as soon as the half's softmax warps
//     have read S / dP into registers, and a tile's dQ product during the next
//     tile; otherwise each half's products follow its softmax.
//   warps 0-3 / 4-7 (half 0 / 1): read S^T_h and dP^T_h from TMEM, form
//       P^T = exp2(S^T scale log2e - lse log2e) (masked) and
//       dS^T = P^T (dP^T - D) in packed fp32 pairs, write P^T as bf16 into
//       TMEM and dS^T as bf16 into the swizzled shared-memory tile.  Then each
//       warpgroup adds half of the previous tile's dQ columns (thread t: query
//       t) into global dq: staged in shared memory, one TMA tensor reduce-add
//       (cp.reduce.async.bulk.tensor .add) per warp.  At the end warps 0-3
//       store dK (times scale) and the first half of dV's columns, warps 4-7
//       the second half.
// 10 warps, so that a thread may hold 168 registers.
//
// TMEM columns: [0,64) S^T_0, [64,128) dP^T_0, [128,192) S^T_1,
// [192,256) dP^T_1, then dV (d_v), dK (r), dQ (r), and where they fit P^T_0,
// P^T_1 (32 columns each; otherwise P^T_h sits in the first 32 of S^T_h).
// At r = 128, dV, dK and dQ do not fit beside the score tiles: dQ_i is then
// computed over S^T_1 / dP^T_1 once the half-1 softmax has consumed them,
// warps 4-7 read it back at once, and the next half-1 scores follow.
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
constexpr int kTcThreads = 320;    // 2 x 4 softmax warps, the MMA warp, the TMA warp
constexpr int kTmemColsTc = 512;
constexpr int kBoxB = 128 * 128;   // one 64-column (128-byte) box of a 128-row tile

constexpr int align1k(int x) { return (x + 1023) / 1024 * 1024; }

template <int R, int DV>
struct TCfg {
  // Q / K rows are r bf16 = 2r bytes: one swizzle span of min(2r, 128) bytes,
  // in QK_NBOX boxes of QK_BOXW columns (two 128-byte boxes at r = 128)
  static constexpr int QK_SW = 2 * R < 128 ? 2 * R : 128;
  static constexpr int QK_NBOX = 2 * R / QK_SW;
  static constexpr int QK_BOXW = QK_SW / 2;
  static constexpr uint32_t QK_LAYOUT = QK_SW == 32 ? 6u : (QK_SW == 64 ? 4u : 2u);
  static constexpr int KSTEP_PER_BOX = QK_SW / 32;  // 16-column K steps per box
  static constexpr int KBOX = kKeys * QK_SW;        // one box of the K tile
  static constexpr int KB = QK_NBOX * KBOX;         // K tile
  static constexpr int VB = kKeys * DV * 2;         // V tile (DV / 64 boxes)
  // Q / dO arrive in 64-query half tiles through a ring of slots: a slot is
  // released as soon as its half's dV / dK products have read it
  static constexpr int QHBOX = kHalfQ * QK_SW;      // one box of a Q half tile
  static constexpr int QHB = QK_NBOX * QHBOX;       // Q half tile
  static constexpr int OHB = kHalfQ * DV * 2;       // dO half tile (DV / 64 boxes)
  static constexpr int OBOX = kHalfQ * 128;         // one 64-column box of a dO half tile
  static constexpr int SL_Q = 0, SL_O = align1k(QHB), SL_L = SL_O + OHB, SL_D = SL_L + kHalfQ * 4;
  static constexpr int SLOT = align1k(SL_D + kHalfQ * 4);
  static constexpr int DSB = kKeys * kQT * 2;       // dS^T tile: [2 halves][128 keys][64 queries]
  // dQ of a tile in TMEM: in columns of its own where they fit (r <= 64), else
  // over S^T_1 / dP^T_1 once the half-1 softmax has consumed them (r = 128)
  static constexpr bool DQ_OWN = 256 + DV + 2 * R <= kTmemColsTc;
  // dQ read back and staged for the TMA reduce-add, boxes of DQ_W fp32
  // columns x 32 rows (one per warp) swizzled over DQ_SW bytes: with its own
  // columns each softmax warpgroup takes R / 2 columns after the next tile's
  // softmax; over S^T_1 / dP^T_1, warps 4-7 take all R at once, right after
  // their softmax, and stage them 32 columns at a time
  static constexpr int DQ_W = DQ_OWN ? R / 2 : 32;
  static constexpr int DQ_SW = DQ_W * 4;
  static constexpr int DQ_LAYOUT_SHIFT = DQ_SW == 128 ? 0 : (DQ_SW == 64 ? 1 : 2);
  static constexpr int DQB = DQ_OWN ? kQT * R * 4 : 4 * 32 * DQ_SW;
  static constexpr int OFF_K = 0;
  static constexpr int OFF_V = align1k(KB);
  static constexpr int OFF_SL = OFF_V + VB;
  // without the dS tiles: K, V, a ring of n slots, the dQ stage, barriers, alignment slack
  static constexpr int fixed(int n) { return OFF_SL + n * SLOT + DQB + 256 + 1024; }
  static constexpr int NDS = fixed(4) + 2 * DSB <= 227 * 1024 ? 2 : 1;   // dS^T tiles in flight
  // half-tile slots: 4 (a fifth, where it fits, measured slower), 3 where 4 do not fit
  static constexpr int NSLOT = fixed(4) + NDS * DSB <= 227 * 1024 ? 4 : 3;
  static constexpr int OFF_DS = OFF_SL + NSLOT * SLOT;
  static constexpr int OFF_DQ = OFF_DS + NDS * DSB;
  static constexpr int OFF_BAR = OFF_DQ + DQB;
  // at least 116 KB so that one CTA (and its 512 TMEM columns) sits on an SM alone
  static constexpr int SMEM = std::max(OFF_BAR + 256 + 1024, 116 * 1024);
  static_assert(OFF_BAR + 256 + 1024 <= 227 * 1024, "shared memory");
  // TMEM columns
  static constexpr int T_S = 0;          // + 128 h: S^T_h
  static constexpr int T_DP = 64;        // + 128 h: dP^T_h
  static constexpr int T_DV = 256, T_DK = 256 + DV, T_DQ = DQ_OWN ? 256 + DV + R : 128;
  static_assert(T_DK + R <= kTmemColsTc && (!DQ_OWN || T_DQ + R <= kTmemColsTc), "TMEM columns");
  static constexpr bool P_OWN = DQ_OWN && T_DQ + R + 2 * (kHalfQ / 2) <= kTmemColsTc;  // P^T in columns of its own
  static constexpr int T_P = P_OWN ? T_DQ + R : T_S;   // + (P_OWN ? 32 : 128) h: P^T_h
  static constexpr int P_STRIDE = P_OWN ? kHalfQ / 2 : 128;
  // With P^T in its own columns and two dS tiles, the next tile's scores of a
  // half are issued as soon as the half's softmax warps have read S / dP into
  // registers, and a tile's dQ product one step later; otherwise the products
  // follow the softmax of each half.
  static constexpr bool EARLY = P_OWN && NDS == 2;
  // instruction descriptors
  static constexpr uint32_t ID_S = instr_desc(kKeys, kHalfQ, false);       // S^T, dP^T
  static constexpr uint32_t ID_DV = instr_desc(kKeys, DV, true);           // A = P^T (TMEM), B = dO MN-major
  static constexpr uint32_t ID_DK = instr_desc(kKeys, R, true);            // A = dS^T K-major, B = Q MN-major
  static constexpr uint32_t ID_DQ = instr_desc(kQT, R, true, true);        // A = dS MN-major, B = K MN-major
};

struct TcMaps {
  CUtensorMap q, k, v, d_out, dq;
};

// TMA tensor reduce-add of a shared-memory box into global memory (bulk group).
__device__ __forceinline__ void tma_reduce_add_3d(const CUtensorMap* map, const void* src, int x, int y, int z) {
  asm volatile(
      "cp.reduce.async.bulk.tensor.3d.global.shared::cta.add.tile.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(smem_addr(src)), "r"(x), "r"(y), "r"(z)
      : "memory");
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
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t* v) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : TK_R8(0)
      : "r"(taddr)
      : "memory");
}
// N consecutive 32-bit columns (N = 8, 16, 32 or 64).
template <int N>
__device__ __forceinline__ void tmem_ld_n(uint32_t taddr, uint32_t* v) {
  if constexpr (N == 8) tmem_ld8(taddr, v);
  else if constexpr (N == 16) tmem_ld16(taddr, v);
  else if constexpr (N == 32) tmem_ld32(taddr, v);
  else tmem_ld64(taddr, v);
}

__device__ __forceinline__ uint32_t pack2(float2 x) {
  __nv_bfloat162 v = __floats2bfloat162_rn(x.x, x.y);  // low half = x.x
  return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ float2 f2(uint32_t a, uint32_t b) {
  return make_float2(__uint_as_float(a), __uint_as_float(b));
}

// N TMEM columns (fp32) of this thread's lane, times `mul`, to dst (16-byte aligned).
template <int N>
__device__ __forceinline__ void tmem_rows_out(uint32_t taddr, float* dst, float mul, bool store) {
#pragma unroll
  for (int c0 = 0; c0 < N; c0 += 32) {
    constexpr int W = N < 32 ? N : 32;
    uint32_t v[W];
    tmem_ld_n<W>(taddr + c0, v);
    if (store) {
#pragma unroll
      for (int c = 0; c < W / 4; ++c)
        reinterpret_cast<float4*>(dst + c0)[c] =
            make_float4(__uint_as_float(v[4 * c]) * mul, __uint_as_float(v[4 * c + 1]) * mul,
                        __uint_as_float(v[4 * c + 2]) * mul, __uint_as_float(v[4 * c + 3]) * mul);
    }
  }
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
  uint64_t* sl_full = bars + 1;      // [NSLOT] half-tile slot loaded
  uint64_t* sl_empty = bars + 6;     // [NSLOT] half-tile slot consumed
  uint64_t* s_full = bars + 11;      // [2] S^T_h, dP^T_h in TMEM
  uint64_t* p_ready = bars + 13;     // [2] P^T_h in TMEM, dS^T_h in shared memory
  uint64_t* p_free = bars + 15;      // [2] P^T_h read by the dV product (P in its own columns)
  uint64_t* ds_free = bars + 17;     // [NDS] dS^T tile read by its last product
  uint64_t* dq_full = bars + 19;
  uint64_t* dq_empty = bars + 20;
  uint64_t* acc_full = bars + 21;
  uint64_t* s_free = bars + 22;      // [2] S^T_h, dP^T_h read into registers (EARLY schedule)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 24);

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
  // half tile u = 2 t + h lives in slot u % NSLOT, its (u / NSLOT)-th use of the slot
  auto slot_of = [](int t, int h) { return (2 * t + h) % C::NSLOT; };
  auto slot_par = [](int t, int h) { return static_cast<uint32_t>(((2 * t + h) / C::NSLOT) & 1); };

  if (tid == 0) {
    mbar_init(kv_full, 1);
    for (int s = 0; s < C::NSLOT; ++s) {
      mbar_init(&sl_full[s], 1);
      mbar_init(&sl_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&s_full[s], 1);
      mbar_init(&p_ready[s], 128);
      mbar_init(&p_free[s], 1);
      mbar_init(&s_free[s], 128);
    }
    for (int s = 0; s < NDS; ++s) mbar_init(&ds_free[s], 1);
    mbar_init(dq_full, 1);
    mbar_init(dq_empty, C::DQ_OWN ? 256 : 128);
    mbar_init(acc_full, 1);
    fence_barrier_init();
  }
  if (warp == 8) {
    tmem_alloc(tmem_slot, kTmemColsTc);
    tmem_relinquish();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 9) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0) {
      const int kv_plane = b * p.Hkv + g;
      prefetch_map(&maps.q);
      prefetch_map(&maps.k);
      prefetch_map(&maps.v);
      prefetch_map(&maps.d_out);
      mbar_arrive_expect_tx(kv_full, C::KB + C::VB);
      for (int x = 0; x < C::QK_NBOX; ++x)
        tma_load_3d(smem + C::OFF_K + x * C::KBOX, &maps.k, x * C::QK_BOXW, j * kKeys, kv_plane, kv_full);
      for (int x = 0; x < DV / 64; ++x)
        tma_load_3d(smem + C::OFF_V + x * kBoxB, &maps.v, 64 * x, j * kKeys, kv_plane, kv_full);
      int issued = 0;
      for (int u = 0; u < 2 * n_tiles; ++u) {
        const int sl = u % C::NSLOT;
        if (u >= C::NSLOT && !mbar_wait(&sl_empty[sl], ((u / C::NSLOT) - 1) & 1, p.err)) break;
        const int t = u >> 1, h = u & 1;
        const int bh = b * p.Hq + tile_head(t), row = tile_q(t) * kQT + h * kHalfQ;
        unsigned char* sb = smem + C::OFF_SL + sl * C::SLOT;
        mbar_arrive_expect_tx(&sl_full[sl], C::QHB + C::OHB + 2 * kHalfQ * 4);
        for (int x = 0; x < C::QK_NBOX; ++x)
          tma_load_3d(sb + C::SL_Q + x * C::QHBOX, &maps.q, x * C::QK_BOXW, row, bh, &sl_full[sl]);
        for (int x = 0; x < DV / 64; ++x)
          tma_load_3d(sb + C::SL_O + x * C::OBOX, &maps.d_out, 64 * x, row, bh, &sl_full[sl]);
        const size_t srow = static_cast<size_t>(bh) * p.S_pad + row;
        bulk_g2s(sb + C::SL_L, p.nl2 + srow, kHalfQ * 4, &sl_full[sl]);
        bulk_g2s(sb + C::SL_D, p.nd + srow, kHalfQ * 4, &sl_full[sl]);
        issued = u + 1;
      }
      // no copy may still be landing in shared memory when the CTA exits
      // (normally all were consumed; after a timed-out wait, bounded waits)
      mbar_wait(kv_full, 0, p.err);
      for (int u = std::max(0, issued - C::NSLOT); u < issued; ++u)
        mbar_wait(&sl_full[u % C::NSLOT], (u / C::NSLOT) & 1, p.err);
    }
  } else if (warp == 8) {
    // ------------------------------------------------------------------ MMA issuer
    const uint32_t s_base = smem_addr(smem);
    // one descriptor serves a tile read K-major and MN-major: SBO is the stride of
    // 8-row groups either way, LBO the stride of MN atoms (unused when N fits one)
    const Desc dK_d = make_desc(s_base + C::OFF_K, C::KBOX, 8 * C::QK_SW, C::QK_LAYOUT);  // K
    const Desc dV_a = make_desc(s_base + C::OFF_V, 16, 1024, 2u);                         // V, K-major
    const Desc dQ_b = make_desc(s_base + C::OFF_SL + C::SL_Q, C::QHBOX, 8 * C::QK_SW, C::QK_LAYOUT);  // Q_h
    const Desc dO_bk = make_desc(s_base + C::OFF_SL + C::SL_O, 16, 1024, 2u);             // dO_h, K-major
    const Desc dO_bm = make_desc(s_base + C::OFF_SL + C::SL_O, C::OBOX, 1024, 2u);        // dO_h, MN-major
    const Desc dS_ak = make_desc(s_base + C::OFF_DS, 16, 1024, 2u);                       // dS^T, K-major
    const Desc dS_am = make_desc(s_base + C::OFF_DS, C::DSB / 2, 1024, 2u);               // dS, MN-major
    auto issue_sdp = [&](int t, int h) {   // S^T_h, dP^T_h of tile t
      const uint32_t so = slot_of(t, h) * C::SLOT;
#pragma unroll
      for (int k = 0; k < R / 16; ++k) {
        const uint32_t kb = (k / C::KSTEP_PER_BOX), ko = (k % C::KSTEP_PER_BOX) * 32;
        mma_ss_e(tmem + C::T_S + 128 * h, dK_d.at(kb * C::KBOX + ko), dQ_b.at(so + kb * C::QHBOX + ko), C::ID_S,
                 k > 0);
      }
#pragma unroll
      for (int k = 0; k < DV / 16; ++k)
        mma_ss_e(tmem + C::T_DP + 128 * h, dV_a.at((k / 4) * kBoxB + (k % 4) * 32),
                 dO_bk.at(so + (k / 4) * C::OBOX + (k % 4) * 32), C::ID_S, k > 0);
      tc_commit_e(&s_full[h]);
    };
    auto issue_dvdk = [&](int t, int h) {  // dV += P^T_h dO_h, dK += dS^T_h Q_h; the slot is then free
      const uint32_t so = slot_of(t, h) * C::SLOT;
      const uint32_t dso = (t % NDS) * C::DSB + h * (C::DSB / 2);
#pragma unroll
      for (int kk = 0; kk < kHalfQ / 16; ++kk)
        mma_ts_e(tmem + C::T_DV, tmem + C::T_P + C::P_STRIDE * h + 8 * kk, dO_bm.at(so + 16 * kk * 128),
                 C::ID_DV, (t > 0 || h > 0 || kk > 0) ? 1u : 0u);
      if (C::P_OWN) tc_commit_e(&p_free[h]);
#pragma unroll
      for (int kk = 0; kk < kHalfQ / 16; ++kk)
        mma_ss_e(tmem + C::T_DK, dS_ak.at(dso + kk * 32), dQ_b.at(so + 16 * kk * C::QK_SW), C::ID_DK,
                 (t > 0 || h > 0 || kk > 0) ? 1u : 0u);
      tc_commit_e(&sl_empty[slot_of(t, h)]);
    };
    auto issue_dq = [&](int t) {           // dQ_t = dS K over the 128 keys
      const uint32_t dso = (t % NDS) * C::DSB;
#pragma unroll
      for (int k = 0; k < kKeys / 16; ++k)
        mma_ss_e(tmem + C::T_DQ, dS_am.at(dso + k * 16 * 128), dK_d.at(k * 16 * C::QK_SW), C::ID_DQ, k > 0);
      tc_commit_e(dq_full);
      tc_commit_e(&ds_free[t % NDS]);
    };
    auto wait_all = [&](uint64_t* bar, uint32_t parity) {
      return __all_sync(0xffffffffu, mbar_wait(bar, parity, p.err));
    };
    bool ok = wait_all(kv_full, 0) && wait_all(&sl_full[0], 0);
    if (ok) {
      tc_fence_after();
      issue_sdp(0, 0);
      ok = wait_all(&sl_full[1], 0);
      tc_fence_after();
      if (ok) issue_sdp(0, 1);
    }
    if constexpr (C::EARLY) {
      // per tile and half: the next tile's scores as soon as the half's softmax
      // warps release S / dP, then (half 0) the previous tile's dQ product, then
      // this tile's dV / dK products when P / dS arrive
      for (int t = 0; ok && t < n_tiles; ++t) {
        for (int h = 0; ok && h < 2; ++h) {
          if (t + 1 < n_tiles) {
            if (!(ok = wait_all(&s_free[h], t & 1) && wait_all(&sl_full[slot_of(t + 1, h)], slot_par(t + 1, h))))
              break;
            tc_fence_after();
            issue_sdp(t + 1, h);
          }
          if (h == 0 && t > 0) {
            if (t > 1 && !(ok = wait_all(dq_empty, (t - 2) & 1))) break;
            tc_fence_after();
            issue_dq(t - 1);
          }
          if (!(ok = wait_all(&p_ready[h], t & 1))) break;
          tc_fence_after();
          issue_dvdk(t, h);
        }
      }
      if (ok && n_tiles > 1) ok = wait_all(dq_empty, (n_tiles - 2) & 1);
      if (ok) {
        tc_fence_after();
        issue_dq(n_tiles - 1);
      }
    } else {
      for (int t = 0; ok && t < n_tiles; ++t) {
        const bool next = t + 1 < n_tiles;
        for (int h = 0; ok && h < 2; ++h) {
          if (!(ok = wait_all(&p_ready[h], t & 1))) break;
          if (next && !(ok = wait_all(&sl_full[slot_of(t + 1, h)], slot_par(t + 1, h)))) break;
          tc_fence_after();
          // P^T_h in columns of its own: the next tile's scores of this half go
          // first; otherwise P^T_h overlays S^T_h and its dV product goes first
          if (C::P_OWN && next) issue_sdp(t + 1, h);
          issue_dvdk(t, h);
          if (h == 1) {
            // dQ before the next tile's half-1 scores: with one dS tile the next
            // tile's half-0 dS waits for it, and without columns of its own dQ
            // occupies S^T_1 / dP^T_1 until warps 4-7 have read it
            if (C::DQ_OWN && t > 0 && !(ok = wait_all(dq_empty, (t - 1) & 1))) break;
            tc_fence_after();
            issue_dq(t);
            if (!C::DQ_OWN && next) {
              if (!(ok = wait_all(dq_empty, t & 1))) break;
              tc_fence_after();
            }
          }
          if (!C::P_OWN && next) issue_sdp(t + 1, h);
        }
      }
    }
    if (ok) tc_commit_e(acc_full);
  } else {
    // ------------------------------------------------------------------ softmax gradient warps
    const int h = warp >> 2;                      // query half
    const int kt = (warp & 3) * 32 + lane;        // key of this thread within the tile (TMEM lane)
    const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t tS = tmem + C::T_S + 128 * h + lane_off, tD = tmem + C::T_DP + 128 * h + lane_off;
    const uint32_t tP = tmem + C::T_P + C::P_STRIDE * h + lane_off;
    const bool kvalid = j * kKeys + kt < S;
    const float sl2 = p.scale * 1.4426950408889634f;
    const float2 sl2x2 = make_float2(sl2, sl2);
    bool ok = true, pending = false;
    // dQ of tile t (thread kt: query kt of the tile), columns [h R/2, (h+1) R/2):
    // read from TMEM after the next tile's softmax (dq_fetch), then staged in
    // shared memory and added into global dq by a TMA reduce per warp (its 32
    // rows), so that no warp waits for another (dq_store).
    unsigned char* dq_box =
        smem + C::OFF_DQ + (C::DQ_OWN ? h * (kQT * C::DQ_SW) : 0) + (warp & 3) * (32 * C::DQ_SW);
    uint32_t wq[C::DQ_W];
    bool dq_ok = false;
    auto dq_fetch = [&](int t) {
      dq_ok = __all_sync(0xffffffffu, ok && mbar_wait(dq_full, t & 1, p.err));
      if (dq_ok) {
        tc_fence_after();
        tmem_ld_n<C::DQ_W>(tmem + C::T_DQ + h * C::DQ_W + lane_off, wq);
        tc_fence_before();
        mbar_arrive(dq_empty);
      }
    };
    auto dq_store = [&](int t) {
      const int row0 = tile_q(t) * kQT + (warp & 3) * 32;   // first query of this warp's rows
      if (dq_ok && row0 < S) {
        if (lane == 0 && pending) bulk_wait_read_all();   // the previous reduce has read the box
        __syncwarp();
#pragma unroll
        for (int c = 0; c < C::DQ_SW / 16; ++c) {
          const int pc = c ^ ((lane >> C::DQ_LAYOUT_SHIFT) & (C::DQ_SW / 16 - 1));
          *reinterpret_cast<float4*>(dq_box + lane * C::DQ_SW + pc * 16) =
              make_float4(__uint_as_float(wq[4 * c]) * p.scale, __uint_as_float(wq[4 * c + 1]) * p.scale,
                          __uint_as_float(wq[4 * c + 2]) * p.scale, __uint_as_float(wq[4 * c + 3]) * p.scale);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_reduce_add_3d(&maps.dq, dq_box, h * C::DQ_W, row0, b * p.Hq + tile_head(t));
          bulk_commit();
          pending = true;
        }
      }
      if (!dq_ok) ok = false;
      dq_ok = false;
    };
    // r = 128 (dQ over S^T_1 / dP^T_1): warps 4-7 read dQ_t right after their
    // softmax of tile t, 64 columns at a time (the first half staged before the
    // second is read), which then releases S^T_1 / dP^T_1 for the next scores;
    // each half is added into dq DQ_W columns at a time
    auto dq_all = [&](int t) {
      static_assert(C::DQ_OWN || R == 128, "dQ over S^T_1 / dP^T_1 is laid out for r = 128");
      const bool okw = __all_sync(0xffffffffu, ok && mbar_wait(dq_full, t & 1, p.err));
      const int row0 = tile_q(t) * kQT + (warp & 3) * 32;
      if (okw) tc_fence_after();
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        uint32_t w[64];
        if (okw) {
          tmem_ld64(tmem + C::T_DQ + 64 * half + lane_off, w);
          if (half == 1) {
            tc_fence_before();
            mbar_arrive(dq_empty);
          }
        }
        if (okw && row0 < S) {
#pragma unroll
          for (int ps = 0; ps < 64 / C::DQ_W; ++ps) {
            if (lane == 0 && pending) bulk_wait_read_all();   // the previous reduce has read the box
            __syncwarp();
#pragma unroll
            for (int c = 0; c < C::DQ_SW / 16; ++c) {
              const int pc = c ^ ((lane >> C::DQ_LAYOUT_SHIFT) & (C::DQ_SW / 16 - 1));
              const int e = ps * C::DQ_W + 4 * c;
              *reinterpret_cast<float4*>(dq_box + lane * C::DQ_SW + pc * 16) =
                  make_float4(__uint_as_float(w[e]) * p.scale, __uint_as_float(w[e + 1]) * p.scale,
                              __uint_as_float(w[e + 2]) * p.scale, __uint_as_float(w[e + 3]) * p.scale);
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              tma_reduce_add_3d(&maps.dq, dq_box, 64 * half + ps * C::DQ_W, row0, b * p.Hq + tile_head(t));
              bulk_commit();
              pending = true;
            }
          }
        }
      }
      if (!okw) ok = false;
    };
    for (int t = 0; t < n_tiles; ++t) {
      const int sl = slot_of(t, h), buf = t % NDS;
      if (ok) {
        ok = mbar_wait(&s_full[h], t & 1, p.err) && mbar_wait(&sl_full[sl], slot_par(t, h), p.err);
        if (ok && t >= NDS) ok = mbar_wait(&ds_free[buf], ((t / NDS) - 1) & 1, p.err);
        ok = __all_sync(0xffffffffu, ok);
      }
      if (ok) {
        tc_fence_after();
        const unsigned char* sb = smem + C::OFF_SL + sl * C::SLOT;
        const float* nl2 = reinterpret_cast<const float*>(sb + C::SL_L);
        const float* nd = reinterpret_cast<const float*>(sb + C::SL_D);
        unsigned char* ds_row = smem + C::OFF_DS + buf * C::DSB + h * (C::DSB / 2) + kt * 128;
        // keys past S, and keys after the query on the diagonal tile, get weight 0
        const int qlim = (p.causal && tile_q(t) == j) ? kt - h * kHalfQ : 0;  // visible iff column >= qlim
        // warp-uniform choice: both paths issue warp-collective TMEM loads and stores
        const bool masked = __any_sync(0xffffffffu, !kvalid || qlim > 0);
        auto chunk = [&](auto mask_tag, int c) {
          constexpr bool kMask = decltype(mask_tag)::value;
          uint32_t v[64];   // [0, 32): S^T, [32, 64): dP^T
          tmem_ld32x2(tS + 32 * c, tD + 32 * c, v);
          if (C::EARLY && c == kHalfQ / 32 - 1) {   // S^T_h, dP^T_h may be overwritten
            tc_fence_before();
            mbar_arrive(&s_free[h]);
          }
          uint32_t pk[16], dk[16];
#pragma unroll
          for (int e2 = 0; e2 < 16; ++e2) {
            const int col = 32 * c + 2 * e2;
            float2 x = ffma2(f2(v[2 * e2], v[2 * e2 + 1]), sl2x2, *reinterpret_cast<const float2*>(nl2 + col));
            if (kMask) {
              if (!kvalid || col < qlim) x.x = -INFINITY;
              if (!kvalid || col + 1 < qlim) x.y = -INFINITY;
            }
            const float2 pr = make_float2(fast_exp2(x.x), fast_exp2(x.y));
            const float2 dsv = fmul2(pr, fadd2(f2(v[32 + 2 * e2], v[33 + 2 * e2]),
                                               *reinterpret_cast<const float2*>(nd + col)));
            pk[e2] = pack2(pr);
            dk[e2] = pack2(dsv);
          }
          // P^T_h may overwrite the previous tile's only once its dV product has read it
          if (C::P_OWN && c == 0 && t > 0) {
            const bool okp = mbar_wait(&p_free[h], (t - 1) & 1, p.err);
            if (!__all_sync(0xffffffffu, okp)) ok = false;
          }
          tmem_st16(tP + 16 * c, pk);
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
      if constexpr (C::DQ_OWN) {
        if (t > 0) {
          dq_fetch(t - 1);
          dq_store(t - 1);
        }
      } else if (h == 1) {
        dq_all(t);
      }
    }
    if (C::DQ_OWN && n_tiles > 0) {
      dq_fetch(n_tiles - 1);
      dq_store(n_tiles - 1);
    }
    if (pending) bulk_wait_all();
    if (ok) ok = mbar_wait(acc_full, 0, p.err);
    if (__all_sync(0xffffffffu, ok)) {
      tc_fence_after();
      const int key = j * kKeys + kt;
      const size_t kx = (static_cast<size_t>(b) * p.Hkv + g) * S + key;
      const bool store = key < S;
      if (h == 0) {
        tmem_rows_out<R>(tmem + C::T_DK + lane_off, p.dk + kx * R, p.scale, store);
        tmem_rows_out<DV / 2>(tmem + C::T_DV + lane_off, p.dv + kx * DV, 1.f, store);
      } else {
        tmem_rows_out<DV / 2>(tmem + C::T_DV + DV / 2 + lane_off, p.dv + kx * DV + DV / 2, 1.f, store);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 8) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemColsTc);
  }
}

template <int R, int DV>
cudaError_t launch_tc(const BackwardParams& p, cudaStream_t stream) {
  using C = TCfg<R, DV>;
  TcMaps maps;
  if (!make_map(&maps.q, p.q, R, p.S, p.B * p.Hq, C::QK_BOXW, kHalfQ, C::QK_SW) ||
      !make_map(&maps.k, p.k, R, p.S, p.B * p.Hkv, C::QK_BOXW, kKeys, C::QK_SW) ||
      !make_map(&maps.v, p.v, DV, p.S, p.B * p.Hkv, 64, kKeys, 128) ||
      !make_map(&maps.d_out, p.d_out, DV, p.S, p.B * p.Hq, 64, kHalfQ, 128) ||
      !make_map(&maps.dq, p.dq, R, p.S, p.B * p.Hq, C::DQ_W, 32, C::DQ_SW, true))
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
    case 128: return tc_by_dv<128>(p, stream, unsupported);
  }
  *unsupported = 1;
  return cudaSuccess;
}

}  // namespace tk
