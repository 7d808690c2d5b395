// Causal (or full) prefill attention with thin keys on the 5th-generation
// tensor cores: tcgen05.mma with accumulators in tensor memory (TMEM),
// operands staged in shared memory by TMA.
//
// Paper: Section 2.1, Eqs. 1-4 (softmax(Q K^T * scale) V with r-wide Q, K and
// d_v-wide V); Appendix E (prefill is compute-bound; thin keys cut the Q K^T
// work by d_head / r).
//
// One CTA per SM computes two consecutive 128-row query tiles, A and B, of one
// (sequence, query head); they share every 128-row K / V tile of a TMA ring.
//   warp 8 (one lane): TMA loads of both Q tiles (once) and of the K / V tiles.
//   warp 9 (whole warp, one elected lane issues): per kv tile j, for x in A, B
//       O_x += P_x(j) V_j        (M=128, N=d_v, K=128; P_x(j) read from TMEM,
//                                 in two 64-key halves as the softmax publishes them)
//       S_x(j+1) = Q_x K_{j+1}^T (M=128, N=128, K=r; bf16 in, fp32 in TMEM)
//     signalling completion with tcgen05.commit onto mbarriers, so one tile's
//     softmax overlaps the other tile's matrix products.
//   warps 0-3 / 4-7 (thread i owns query row i = TMEM lane i of tile A / B):
//     read S from TMEM, apply the causal / length mask, keep the running max m
//     and sum l (log2 domain), write P = exp2(S * scale*log2e - m) as bf16 into
//     the first 64 TMEM columns of S, and at the end write O / l.
//   warps 10-11 (int8 / int4 key caches only): widen each K tile's codes to
//     bf16 in the swizzled operand layout, half a tile each.
// The running max is updated lazily: O and l are rescaled only when a tile's
// maximum exceeds the max in use by more than 8 (a factor 256), so the
// weights stay <= 256 and the result is unchanged (O / l uses one consistent
// max).
//
// TMEM columns: [0,128) S_A, [128,256) S_B (each: fp32 scores, the first 64
// columns later hold P as packed bf16 pairs), [256,384) O_A, [384,512) O_B.
#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "tc05.cuh"
#include "widen.cuh"

namespace tk {
namespace {

constexpr int kBM = 128;          // query rows per tile
constexpr int kBN = 128;          // keys per kv tile
constexpr int kThreads = 320;     // 2 x 4 softmax warps, 1 TMA warp, 1 MMA warp
// quantised-key caches add two warps that widen the key codes of each tile
template <int KF>
constexpr int threads_for() { return KF == 0 ? kThreads : kThreads + 64; }
constexpr int kTmemCols = 512;
constexpr float kRescaleThreshold = 8.0f;  // log2 units
// P of a tile is published in kParts key ranges, so the P V products of one
// range run while the softmax computes the next (two halves measured best;
// four add more handoff latency than they hide).
constexpr int kParts = 2;
constexpr int kPartPairs = kBN / 2 / kParts;  // packed bf16 pairs (TMEM columns) per part

// ---------------------------------------------------------------- softmax helpers

__device__ __forceinline__ float max3f(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// Maximum of 128 floats held in registers (three-input max tree, few temporaries).
__device__ __forceinline__ float max128(const uint32_t* v) {
#define TK_F(i) __uint_as_float(v[i])
  float a[16];
#pragma unroll
  for (int i = 0; i < 16; ++i)
    a[i] = max3f(max3f(TK_F(8 * i), TK_F(8 * i + 1), TK_F(8 * i + 2)),
                 max3f(TK_F(8 * i + 3), TK_F(8 * i + 4), TK_F(8 * i + 5)),
                 fmaxf(TK_F(8 * i + 6), TK_F(8 * i + 7)));
#undef TK_F
  const float b0 = max3f(a[0], a[1], a[2]), b1 = max3f(a[3], a[4], a[5]);
  const float b2 = max3f(a[6], a[7], a[8]), b3 = max3f(a[9], a[10], a[11]);
  const float b4 = max3f(a[12], a[13], a[14]);
  return fmaxf(max3f(b0, b1, b2), max3f(b3, b4, a[15]));
}


// Key formats of the cache a chunked prefill reads (the plain prefill is always bf16).
constexpr int kKeyBF16 = 0, kKeyInt8 = 1, kKeyInt4 = 2;

template <int R, int DV, int KF = kKeyBF16>
struct PCfg {
  // Q / K rows are r bf16 = 2r bytes: swizzle span = min(2r, 128) bytes; a row
  // wider than 128 bytes is loaded as 128-byte-wide boxes.
  static constexpr int QK_SW = (2 * R < 128) ? 2 * R : 128;
  static constexpr int QK_BOX = QK_SW / 2;           // elements per box row
  static constexpr int QK_NBOX = (2 * R) / QK_SW;    // boxes per tile
  static constexpr int QK_BOXB = kBM * QK_SW;        // bytes per box
  static constexpr uint32_t QK_LAYOUT = QK_SW == 32 ? 6u : (QK_SW == 64 ? 4u : 2u);
  static constexpr int KSTEP_PER_BOX = QK_SW / 32;   // 16-element K steps per box
  static constexpr int QB = kBM * R * 2;
  static constexpr int KB = kBN * R * 2;
  static constexpr int VB = kBN * DV * 2;
  static constexpr int V_NBOX = DV / 64;             // 128-byte-wide boxes of V
  static constexpr int V_BOXB = kBN * 128;
  // quantised keys: a tile's codes (r or r/2 bytes per key) land in a staging
  // area of the stage, and its 128 fp32 key scales after them
  static constexpr int CODE_ROWB = KF == kKeyInt8 ? R : (KF == kKeyInt4 ? R / 2 : 0);
  static constexpr int STGB = kBN * CODE_ROWB;
  static constexpr int SCB = KF == kKeyBF16 ? 0 : kBN * 4;
  static constexpr int QBA = (QB + 1023) / 1024 * 1024;  // one Q tile, 1 KB aligned
  static constexpr int OFF_Q = 0;                        // two Q tiles
  static constexpr int OFF_K = 2 * QBA;
  static constexpr int KBA = (KB + 1023) / 1024 * 1024;
  static constexpr int STAGE = KBA + VB;
  static constexpr int NST = (2 * QBA + 3 * (STAGE + SCB) + 2 * STGB + 2048 <= 200 * 1024) ? 3 : 2;
  // raw codes wait in a staging slot until the widening warps have widened
  // them: one slot per stage where shared memory allows, else two slots that
  // the TMA warp reuses once they are free; the scales keep one slot per stage
  static constexpr int NSTG = (2 * QBA + NST * (STAGE + SCB + STGB) + 2048 <= 200 * 1024) ? NST : 2;
  static constexpr int OFF_STG = OFF_K + NST * STAGE;
  static constexpr int OFF_SC = OFF_STG + NSTG * STGB;
  static constexpr int OFF_BAR = OFF_SC + NST * SCB;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;      // + slack to align the base to 1 KB
  static_assert(SMEM <= 227 * 1024, "shared memory");
  static constexpr uint32_t IDESC_S = instr_desc(kBM, kBN, false);
  static constexpr uint32_t IDESC_O = instr_desc(kBM, DV, true);
};

// Byte offset, inside a K tile, of the 16-byte piece holding elements e0 .. e0+7
// (e0 a multiple of 8) of key `row`, in the layout the TMA writes with the
// tile's swizzle: box e0 / QK_BOX, row pitch QK_SW bytes, and the piece's index
// within its row XORed with address bits 7.. (32-, 64- or 128-byte swizzle).
template <class C>
__device__ __forceinline__ uint32_t k_piece_offset(int row, int e0) {
  const uint32_t o = static_cast<uint32_t>(row * C::QK_SW + (e0 % C::QK_BOX) * 2);
  constexpr uint32_t mask = static_cast<uint32_t>(C::QK_SW / 16 - 1) << 4;
  return static_cast<uint32_t>((e0 / C::QK_BOX) * C::QK_BOXB) + (o ^ ((o >> 3) & mask));
}

struct Maps {
  CUtensorMap q, k, v;
};

// One CTA (one per SM) computes two consecutive 128-row query tiles, A and B,
// of one (sequence, query head).  They share every K/V tile of the ring, and
// the MMA warp interleaves them so that one tile's softmax overlaps the other
// tile's matrix products:
//   S_A(0) S_B(0) | PV_A(0) S_A(1) PV_B(0) S_B(1) | PV_A(1) S_A(2) PV_B(1) ...
// TMEM columns: [0,128) S_A (P_A in its first 64 columns), [128,256) S_B,
// [256,384) O_A, [384,512) O_B.
//   warps 0-3: softmax and epilogue of tile A (thread i owns row i = TMEM lane i)
//   warps 4-7: the same for tile B
//   warp 8: TMA producer (Q tiles once, K/V tiles into an NST-stage ring)
//   warp 9: MMA issuer
template <int R, int DV, int KF>
__global__ void __launch_bounds__(threads_for<KF>(), 1)
prefill_kernel(const __grid_constant__ Maps maps, const PrefillParams p) {
  using C = PCfg<R, DV, KF>;
  constexpr int NST = C::NST;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* q_full = bars + 0;
  uint64_t* k_full = bars + 1;                  // [NST]
  uint64_t* v_full = k_full + NST;              // [NST]
  uint64_t* kv_empty = v_full + NST;            // [NST]
  uint64_t* s_full = kv_empty + NST;            // [2] (tile A, tile B)
  uint64_t* p_full = s_full + 2;                // [tile][part]: P of one key range
  uint64_t* o_full = p_full + 2 * kParts;       // [2]
  uint64_t* c_full = o_full + 2;                // [NST] cached mode: raw K tile (+ scales) landed
  uint64_t* stg_free = c_full + NST;            // [NSTG] quantised keys: staging slot widened
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(stg_free + C::NSTG);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n_qt = (p.S + kBM - 1) / kBM;
  const int n_tp = (n_qt + 1) / 2;              // query tile pairs
  const int BH = p.B * p.Hq;
  // CTA order: heads in groups of p.head_group whose K/V stay in L2 together;
  // inside a group the heaviest (latest) tile pairs first.
  const int grp = static_cast<int>(blockIdx.x / (p.head_group * n_tp));
  const int rem = static_cast<int>(blockIdx.x - static_cast<long>(grp) * p.head_group * n_tp);
  const int gsize = min(p.head_group, BH - grp * p.head_group);
  const int tp = n_tp - 1 - rem / gsize;
  const int bh = grp * p.head_group + rem % gsize;
  const int b = bh / p.Hq, h = bh % p.Hq;
  const int kv_plane = b * p.Hkv + h / (p.Hq / p.Hkv);
  const int qa = 2 * tp, qb = 2 * tp + 1;
  const bool has_b = qb < n_qt;
  // keys: the sequence's first kv_len cache tokens; query row i sits at position L0 + i
  int L0 = 0;
  if (p.seq_lens) {
    L0 = p.seq_lens[b];
    if (L0 < 0 || L0 > p.kv_limit - p.S) {
      if (tid == 0) record_error(p.err, TK_DEVERR_INDEX);
      L0 = L0 < 0 ? 0 : p.kv_limit - p.S;
    }
  }
  const int kv_len = L0 + p.S;
  const int n_kv_all = (kv_len + kBN - 1) / kBN;
  // a causal query tile needs the kv tiles up to its last row's position
  auto tiles_for = [&](int qt) {
    const int last = L0 + min(qt * kBM + kBM, p.S) - 1;
    return p.causal ? min(n_kv_all, last / kBN + 1) : n_kv_all;
  };
  const int n_a = tiles_for(qa);
  const int n_b = has_b ? tiles_for(qb) : 0;
  const int n_kv = max(n_a, n_b);

  if (tid == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < NST; ++s) {
      // quantised keys: both widening warps arrive on k_full; otherwise the TMA warp
      mbar_init(&k_full[s], KF == kKeyBF16 ? 1 : 2);
      mbar_init(&v_full[s], 1);
      mbar_init(&kv_empty[s], 1);
      mbar_init(&c_full[s], 1);
    }
    for (int s = 0; s < C::NSTG; ++s) mbar_init(&stg_free[s], 2);
    for (int x = 0; x < 2; ++x) {
      mbar_init(&s_full[x], 1);
      for (int h = 0; h < kParts; ++h) mbar_init(&p_full[kParts * x + h], 128);
      mbar_init(&o_full[x], 1);
    }
    fence_barrier_init();
  }
  if (warp == 8) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // A tile is "relayed" when it must be finished in shared memory before the MMA
  // warp may read it: every tile of a quantised cache (codes widened to bf16,
  // by the two widening warps) and, in cached mode, the tile holding the
  // context's end (value rows past it zeroed by the TMA warp: the cache may hold
  // anything there, and 0 * NaN would spread).  Other tiles go straight from the
  // TMA to k_full.
  const bool relay = p.seq_lens != nullptr;
  auto relayed = [&](int j) {
    return relay && (KF != kKeyBF16 || kv_len - j * kBN < kBN);
  };
  // finish(j, part, nparts) of a relayed tile, by warp `part` of the nparts
  // warps that share it: widen its share of the codes, zero its share of the
  // value rows past the context, then publish on k_full (nparts arrivals)
  auto finish = [&](int j, int part, int nparts) -> bool {
    const int st = j % NST;
    unsigned char* sk = smem + C::OFF_K + st * C::STAGE;
    unsigned char* sv = sk + C::KBA;
    // quantised caches use c_full on every tile; a bf16 cache only on its last
    const uint32_t phc = KF != kKeyBF16 ? (j / NST) & 1 : 0;
    bool okc = mbar_wait(&c_full[st], phc, p.err);
    const int n_valid = kv_len - j * kBN;
    if (n_valid < kBN) okc = mbar_wait(&v_full[st], (j / NST) & 1, p.err) && okc;
    if (!__all_sync(0xffffffffu, okc)) return false;
    if constexpr (KF != kKeyBF16) {
      const unsigned char* stg = smem + C::OFF_STG + (j % C::NSTG) * C::STGB;
      constexpr int PPR = R / 8;  // 16-byte bf16 pieces per key row
#pragma unroll 4
      for (int c = part * 32 + lane; c < kBN * PPR; c += 32 * nparts) {
        const int row = c / PPR, e0 = (c % PPR) * 8;
        // exact widening by integer moves (no int-to-float conversions, which
        // would share the ex2 unit with the softmax warps)
        uint4 o;
        if constexpr (KF == kKeyInt8) {
          const uint2 w = *reinterpret_cast<const uint2*>(stg + row * C::CODE_ROWB + e0);
          i8x4_to_bf16(w.x, o.x, o.y);
          i8x4_to_bf16(w.y, o.z, o.w);
        } else {
          const uint32_t w = *reinterpret_cast<const uint32_t*>(stg + row * C::CODE_ROWB + e0 / 2);
          i4x8_to_bf16(w, o.x, o.y, o.z, o.w);
        }
        *reinterpret_cast<uint4*>(sk + k_piece_offset<C>(row, e0)) = o;
      }
    }
    if (n_valid < kBN) {
      const int first = max(n_valid, 0);
      const int per_box = (kBN - first) * 8;   // 16-byte pieces per value box
      for (int c = part * 32 + lane; c < per_box * C::V_NBOX; c += 32 * nparts) {
        const int box = c / per_box, rem2 = c % per_box;
        *reinterpret_cast<uint4*>(sv + box * C::V_BOXB + (first + rem2 / 8) * 128 + (rem2 % 8) * 16) =
            make_uint4(0u, 0u, 0u, 0u);
      }
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    __syncwarp();
    if (lane == 0) {
      mbar_arrive(&k_full[st]);
      if constexpr (KF != kKeyBF16) mbar_arrive(&stg_free[j % C::NSTG]);  // staging slot read
    }
    return true;
  };

  if (warp == 8) {
    // ------------------------------------------------------------------ TMA producer
    // K/V maps are [planes][rows][width]: plane b*Hkv + g with rows = S (plain) or
    // the capacity (contiguous cache), or plane page*Hkv + g with rows = page_size
    // (paged); a 128-key tile is one box, or 128 / page_size boxes from several pages.
    const int g = h / (p.Hq / p.Hkv);
    const int bps = (p.page_size == 0 || p.page_size >= kBN) ? kBN : p.page_size;
    const int nsub = kBN / bps;
    if (lane == 0) {
      prefetch_map(&maps.q);
      prefetch_map(&maps.k);
      prefetch_map(&maps.v);
      mbar_arrive_expect_tx(q_full, has_b ? 2 * C::QB : C::QB);
      for (int x = 0; x < (has_b ? 2 : 1); ++x)
        for (int i = 0; i < C::QK_NBOX; ++i)
          tma_load_3d(smem + C::OFF_Q + x * C::QBA + i * C::QK_BOXB, &maps.q, i * C::QK_BOX,
                      (qa + x) * kBM, bh, q_full);
    }
    // issue(j): wait for the stage, then the TMA loads of tile j
    auto issue = [&](int j) -> bool {
      const int st = j % NST;
      int okw = 1;
      if (j >= NST && lane == 0) okw = mbar_wait(&kv_empty[st], ((j / NST) - 1) & 1, p.err);
      // quantised keys: staging slot j % NSTG must have been widened (tile j - NSTG)
      if (KF != kKeyBF16 && j >= C::NSTG && lane == 0 && okw)
        okw = mbar_wait(&stg_free[j % C::NSTG], ((j / C::NSTG) - 1) & 1, p.err);
      if (!__shfl_sync(0xffffffffu, okw, 0)) return false;
      // lane s < nsub finds the plane and first row of sub-box s
      int plane = kv_plane, row = j * kBN;
      if (p.page_size != 0) {
        const int t = j * kBN + lane * bps;
        int page = -1;  // keys past the sequence's pages read the zero fill
        if (lane < nsub && t < kv_len) {
          page = p.page_table[static_cast<long long>(b) * p.max_pages + (t >> p.page_shift)];
          if (page < 0 || page >= p.num_pages) {
            record_error(p.err, TK_DEVERR_INDEX);
            page = 0;
          }
        }
        plane = page < 0 ? -1 : page * p.Hkv + g;
        row = t & (p.page_size - 1);
      }
      int planes[kBN / 16], rows[kBN / 16];
#pragma unroll
      for (int s2 = 0; s2 < kBN / 16; ++s2) {
        planes[s2] = __shfl_sync(0xffffffffu, plane, s2);
        rows[s2] = __shfl_sync(0xffffffffu, row, s2);
      }
      if (lane == 0) {
        unsigned char* sk = smem + C::OFF_K + st * C::STAGE;
        unsigned char* sv = sk + C::KBA;
        if constexpr (KF == kKeyBF16) {
          uint64_t* kb = relayed(j) ? &c_full[st] : &k_full[st];
          mbar_arrive_expect_tx(kb, C::KB);
          for (int s2 = 0; s2 < nsub; ++s2)
            for (int i = 0; i < C::QK_NBOX; ++i)
              tma_load_3d(sk + i * C::QK_BOXB + s2 * bps * C::QK_SW, &maps.k, i * C::QK_BOX,
                          rows[s2], planes[s2], kb);
        } else {
          // raw codes into staging slot j % NSTG (emptied by the widening warps,
          // waited for above), the tile's key scales into the stage's slot
          unsigned char* stg = smem + C::OFF_STG + (j % C::NSTG) * C::STGB;
          float* sc = reinterpret_cast<float*>(smem + C::OFF_SC + st * C::SCB);
          const int kv0 = j * kBN;
          uint32_t sc_bytes = 0;
          if (p.page_size == 0) {
            sc_bytes = static_cast<uint32_t>(min(kBN, p.capacity - kv0)) * 4u;
          } else {
            for (int s2 = 0; s2 < nsub; ++s2)
              if (planes[s2] >= 0) sc_bytes += static_cast<uint32_t>(bps) * 4u;
          }
          mbar_arrive_expect_tx(&c_full[st], static_cast<uint32_t>(nsub * bps * C::CODE_ROWB) + sc_bytes);
          for (int s2 = 0; s2 < nsub; ++s2)
            tma_load_3d(stg + s2 * bps * C::CODE_ROWB, &maps.k, 0, rows[s2], planes[s2], &c_full[st]);
          if (p.page_size == 0) {
            bulk_g2s(sc, p.k_scale + static_cast<size_t>(kv_plane) * p.capacity + kv0, sc_bytes,
                     &c_full[st]);
          } else {
            for (int s2 = 0; s2 < nsub; ++s2)
              if (planes[s2] >= 0)
                bulk_g2s(sc + s2 * bps,
                         p.k_scale + static_cast<size_t>(planes[s2]) * p.page_size + rows[s2],
                         static_cast<uint32_t>(bps) * 4u, &c_full[st]);
          }
        }
        mbar_arrive_expect_tx(&v_full[st], C::VB);
        for (int s2 = 0; s2 < nsub; ++s2)
          for (int i = 0; i < C::V_NBOX; ++i)
            tma_load_3d(sv + i * C::V_BOXB + s2 * bps * 128, &maps.v, i * 64, rows[s2], planes[s2],
                        &v_full[st]);
      }
      return true;
    };
    if constexpr (KF == kKeyBF16) {
      for (int j = 0; j < n_kv; ++j) {
        if (!issue(j)) break;
        if (relayed(j) && !finish(j, 0, 1)) break;
      }
    } else {
      for (int j = 0; j < n_kv; ++j)
        if (!issue(j)) break;
    }
  } else if (warp >= 10) {
    // ------------------------------------------------------------------ widening warps
    // (quantised keys only): each widens half of every tile's codes
    for (int j = 0; j < n_kv; ++j)
      if (!finish(j, warp - 10, 2)) break;
  } else if (warp == 9) {
    // ------------------------------------------------------------------ MMA issuer
    {
      // descriptors of Q tile A and of the K / V tiles of stage 0; other
      // stages and K steps are start-address offsets from these
      const Desc dq = make_desc(smem_addr(smem + C::OFF_Q), 16, 8 * C::QK_SW, C::QK_LAYOUT);
      const Desc dk = make_desc(smem_addr(smem + C::OFF_K), 16, 8 * C::QK_SW, C::QK_LAYOUT);
      const Desc dv = make_desc(smem_addr(smem + C::OFF_K + C::KBA), C::V_BOXB, 1024, 2u);
      auto issue_s = [&](int x, int st) {  // S_x = Q_x K^T
        const uint32_t qo = x * C::QBA, ko = st * C::STAGE;
#pragma unroll
        for (int k = 0; k < R / 16; ++k) {
          const uint32_t off = (k / C::KSTEP_PER_BOX) * C::QK_BOXB + (k % C::KSTEP_PER_BOX) * 32;
          mma_ss_e(tmem + x * 128, dq.at(qo + off), dk.at(ko + off), C::IDESC_S, k > 0);
        }
        tc_commit_e(&s_full[x]);
      };
      auto issue_pv = [&](int x, int st, bool first, int part) {  // O_x += P_x V, one part
        const uint32_t vo = st * C::STAGE;
        const uint32_t td = tmem + 256 + x * 128, ta = tmem + x * 128;
#pragma unroll
        for (int kk = 0; kk < kBN / 16 / kParts; ++kk) {
          const int k = part * (kBN / 16 / kParts) + kk;
          mma_ts_e(td, ta + 8 * k, dv.at(vo + k * 16 * 128), C::IDESC_O, (!first || k > 0) ? 1u : 0u);
        }
      };
      bool ok = __all_sync(0xffffffffu, mbar_wait(q_full, 0, p.err) && mbar_wait(&k_full[0], 0, p.err));
      if (ok) {
        tc_fence_after();
        issue_s(0, 0);
        if (has_b) issue_s(1, 0);
      }
      for (int j = 0; ok && j < n_kv; ++j) {
        const int st = j % NST;
        const uint32_t ph = (j / NST) & 1;
        const int stn = (j + 1) % NST;
        const uint32_t phn = ((j + 1) / NST) & 1;
        bool v_ready = false;
        for (int x = 0; x < 2 && ok; ++x) {
          const int nx = x == 0 ? n_a : n_b;
          if (j >= nx) continue;
          // each part of P_x(j) feeds its MMAs while the softmax warps compute
          // the next part
          if (!v_ready && !(ok = __all_sync(0xffffffffu, mbar_wait(&v_full[st], ph, p.err)))) break;
          v_ready = true;
          for (int h = 0; ok && h < kParts; ++h) {
            if (!(ok = __all_sync(0xffffffffu, mbar_wait(&p_full[kParts * x + h], j & 1, p.err)))) break;
            tc_fence_after();
            issue_pv(x, st, j == 0, h);
          }
          if (!ok) break;
          if (j + 1 == nx) {
            tc_commit_e(&o_full[x]);
          } else {
            if (!(ok = __all_sync(0xffffffffu, mbar_wait(&k_full[stn], phn, p.err)))) break;
            tc_fence_after();
            issue_s(x, stn);
          }
        }
        if (ok) tc_commit_e(&kv_empty[st]);
      }
    }
  } else {
    // ------------------------------------------------------------------ softmax warps
    const int x = warp >> 2;                   // 0: tile A, 1: tile B
    const int nx = x == 0 ? n_a : n_b;
    const int qt = x == 0 ? qa : qb;
    const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t tS = tmem + x * 128, tO = tmem + 256 + x * 128;
    const int row = qt * kBM + (tid & 127);    // query row of this thread in the chunk
    const int pos = L0 + row;                  // its position among the keys
    const float sl2 = p.scale_log2;
    float m_used = -INFINITY, l = 0.f;
    bool ok = nx > 0;
    for (int j = 0; j < nx; ++j) {
      ok = mbar_wait(&s_full[x], j & 1, p.err);
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      tc_fence_after();
      const int kv0 = j * kBN;
      const bool masked = (p.causal && kv0 + kBN - 1 > L0 + qt * kBM) || (kv0 + kBN > kv_len);
      const int lim = min(kv_len - kv0, p.causal ? pos - kv0 + 1 : kBN);  // visible columns
      // the whole S row of this thread: 128 fp32 scores
      uint32_t v[128];
      tmem_ld128(tS + lane_off, v);
      if constexpr (KF != kKeyBF16) {
        // quantised keys: the products are q . code; each key's fp32 scale turns
        // them into q . k (the scales arrived with the codes on c_full)
        const int st = j % NST;
        if (!__all_sync(0xffffffffu, mbar_wait(&c_full[st], (j / NST) & 1, p.err))) { ok = false; break; }
        const uint32_t sc_addr = smem_addr(smem + C::OFF_SC + st * C::SCB);
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          // volatile loads keep the 32 scale vectors from all being hoisted
          // ahead of their multiplies (128 more live registers: spills)
          float4 f;
          asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                       : "=f"(f.x), "=f"(f.y), "=f"(f.z), "=f"(f.w)
                       : "r"(sc_addr + 16u * i));
          const float2 a = fmul2(make_float2(__uint_as_float(v[4 * i]), __uint_as_float(v[4 * i + 1])),
                                 make_float2(f.x, f.y));
          const float2 c = fmul2(make_float2(__uint_as_float(v[4 * i + 2]), __uint_as_float(v[4 * i + 3])),
                                 make_float2(f.z, f.w));
          v[4 * i] = __float_as_uint(a.x);
          v[4 * i + 1] = __float_as_uint(a.y);
          v[4 * i + 2] = __float_as_uint(c.x);
          v[4 * i + 3] = __float_as_uint(c.y);
        }
      }
      if (masked) {
#pragma unroll
        for (int i = 0; i < 128; ++i)
          if (i >= lim) v[i] = 0xff800000u;  // -inf: masked keys get weight exp2(-inf) = 0
      }
      const float mt = max128(v) * sl2;  // tile max in log2 units (scale > 0)
      const bool resc = mt > m_used + kRescaleThreshold;
      float alpha = 1.f;
      if (resc) {
        alpha = fast_exp2(m_used - mt);   // 0 on the first tile
        m_used = mt;
      }
      l *= alpha;
      // P = exp2(s * scale log2e - m) as bf16 pairs into TMEM columns [0, 64) of S,
      // published in kParts consecutive key ranges
      const float2 sl2x2 = make_float2(sl2, sl2), negm2 = make_float2(-m_used, -m_used);
      float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                       make_float2(0.f, 0.f)};
#pragma unroll
      for (int c = 0; c < kParts; ++c) {
        uint32_t pk[kPartPairs];
#pragma unroll
        for (int i = 0; i < kPartPairs; ++i) {
          const int e = 2 * kPartPairs * c + 2 * i;
          const float2 t = ffma2(make_float2(__uint_as_float(v[e]), __uint_as_float(v[e + 1])),
                                 sl2x2, negm2);
          const float2 pr = make_float2(fast_exp2(t.x), fast_exp2(t.y));
          acc[i & 3] = fadd2(acc[i & 3], pr);
          __nv_bfloat162 b2 = __floats2bfloat162_rn(pr.x, pr.y);  // low half = column e
          pk[i] = *reinterpret_cast<uint32_t*>(&b2);
        }
        tmem_st<kPartPairs>(tS + lane_off + kPartPairs * c, pk);
        if (c == 0 && j > 0 && __any_sync(0xffffffffu, resc)) {
          // O *= alpha before any P V product of this tile accumulates into it; the
          // previous one is complete (the S_j commit covers it)
#pragma unroll 1
          for (int cc = 0; cc < DV / 16; ++cc) {
            uint32_t o[16];
            tmem_ld16(tO + lane_off + 16 * cc, o);
#pragma unroll
            for (int i = 0; i < 16; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
            tmem_st16(tO + lane_off + 16 * cc, o);
          }
        }
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(&p_full[kParts * x + c]);
      }
      const float2 s01 = fadd2(acc[0], acc[1]), s23 = fadd2(acc[2], acc[3]);
      l += (s01.x + s01.y) + (s23.x + s23.y);
    }
    // epilogue: out = O / l
    if (ok) ok = mbar_wait(&o_full[x], 0, p.err);
    if (__all_sync(0xffffffffu, ok)) {
      tc_fence_after();
      const float inv = 1.f / l;
      const bool store = row < p.S;
      const size_t obase = (static_cast<size_t>(bh) * p.S + row) * DV;
      // natural-log logsumexp of the row's scaled scores (for the backward):
      // sum_j exp(scale s_j) = 2^m_used * l
      if (p.lse && store) p.lse[static_cast<size_t>(bh) * p.S + row] = (m_used + log2f(l)) * 0.69314718055994531f;
#pragma unroll
      for (int c = 0; c < DV / 32; ++c) {
        uint32_t v[32];
        tmem_ld32(tO + lane_off + 32 * c, v);
        if (store) {
          if (p.out_f32) {
            float4* dst = reinterpret_cast<float4*>(static_cast<float*>(p.out) + obase + 32 * c);
#pragma unroll
            for (int i = 0; i < 8; ++i)
              dst[i] = make_float4(__uint_as_float(v[4 * i]) * inv, __uint_as_float(v[4 * i + 1]) * inv,
                                   __uint_as_float(v[4 * i + 2]) * inv, __uint_as_float(v[4 * i + 3]) * inv);
          } else {
            uint4* dst = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(p.out) + obase + 32 * c);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              uint32_t w[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                __nv_bfloat162 pr = __floats2bfloat162_rn(__uint_as_float(v[8 * i + 2 * e]) * inv,
                                                          __uint_as_float(v[8 * i + 2 * e + 1]) * inv);
                w[e] = *reinterpret_cast<uint32_t*>(&pr);
              }
              dst[i] = make_uint4(w[0], w[1], w[2], w[3]);
            }
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 8) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------- host side

template <int R, int DV, int KF>
cudaError_t launch_t(const PrefillParams& p, cudaStream_t stream) {
  using C = PCfg<R, DV, KF>;
  Maps maps;
  // K / V: [B*Hkv][S] inputs, a contiguous cache [B*Hkv][capacity] or a paged
  // pool [num_pages*Hkv][page_size] (boxes of min(page_size, 128) rows)
  int kv_rows = p.S, kv_planes = p.B * p.Hkv, box_rows = kBM;
  if (p.seq_lens && p.page_size == 0) {
    kv_rows = p.capacity;
  } else if (p.seq_lens) {
    kv_rows = p.page_size;
    kv_planes = p.num_pages * p.Hkv;
    box_rows = std::min(p.page_size, kBN);
  }
  bool ok = make_map(&maps.q, p.q, R, p.S, p.B * p.Hq, C::QK_BOX, kBM, C::QK_SW) &&
            make_map(&maps.v, p.v, DV, kv_rows, kv_planes, 64, box_rows, 128);
  if constexpr (KF == kKeyBF16)
    ok = ok && make_map(&maps.k, p.k, R, kv_rows, kv_planes, C::QK_BOX, box_rows, C::QK_SW);
  else  // rows of codes, copied as they are into the staging area
    ok = ok && make_map_bytes(&maps.k, p.k, C::CODE_ROWB, kv_rows, kv_planes, box_rows);
  if (!ok) return cudaErrorInvalidValue;
  auto kern = prefill_kernel<R, DV, KF>;
  const int smem = C::SMEM;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const long n_qt = (p.S + kBM - 1) / kBM;
  const long grid = (n_qt + 1) / 2 * p.B * p.Hq;  // one CTA per query tile pair
  PrefillParams pp = p;
  // about 48 MB of K/V per head group
  const long head_bytes = static_cast<long>(p.seq_lens ? p.kv_limit : p.S) * (R + DV) * 2;
  pp.head_group = static_cast<int>(std::max(1L, std::min<long>(p.B * p.Hq, (48L << 20) / head_bytes)));
  if (grid > 0x7fffffffL) return cudaErrorInvalidConfiguration;
  kern<<<static_cast<unsigned>(grid), threads_for<KF>(), smem, stream>>>(maps, pp);
  return cudaGetLastError();
}

template <int R, int DV>
cudaError_t by_kf(const PrefillParams& p, cudaStream_t s, int* uns) {
  // quantised keys only in cached mode (a cache written by the quantising append)
  if (p.k_fmt == kKeyBF16) return launch_t<R, DV, kKeyBF16>(p, s);
  if (!p.seq_lens || !p.k_scale) {
    *uns = 1;
    return cudaSuccess;
  }
  if (p.k_fmt == kKeyInt8) return launch_t<R, DV, kKeyInt8>(p, s);
  if constexpr (R >= 32) {
    if (p.k_fmt == kKeyInt4) return launch_t<R, DV, kKeyInt4>(p, s);
  }
  *uns = 1;
  return cudaSuccess;
}

template <int R>
cudaError_t by_dv(const PrefillParams& p, cudaStream_t s, int* uns) {
  switch (p.DV) {
    case 64: return by_kf<R, 64>(p, s, uns);
    case 128: return by_kf<R, 128>(p, s, uns);
  }
  *uns = 1;
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_prefill(const PrefillParams& p, cudaStream_t stream, int* unsupported) {
  *unsupported = 0;
  switch (p.R) {
    case 16: return by_dv<16>(p, stream, unsupported);
    case 32: return by_dv<32>(p, stream, unsupported);
    case 64: return by_dv<64>(p, stream, unsupported);
    case 128: return by_dv<128>(p, stream, unsupported);
  }
  *unsupported = 1;
  return cudaSuccess;
}

}  // namespace tk
