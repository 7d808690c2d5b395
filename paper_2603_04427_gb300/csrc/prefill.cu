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
// int8 / int4 key caches: key_widen_kernel first widens the context's keys
// once into a contiguous workspace, which the TMA warp then loads like bf16
// keys.  Where shared memory holds two K tiles per stage (r <= 64) each key
// becomes scale * code as the two-term bf16 sum hi + lo
// (|hi + lo - scale * code| <= 2^-17 |scale * code|) and S takes 2r/16 MMA
// steps, Q against hi and then against lo, so the softmax is that of bf16
// keys; otherwise (r = 128) the workspace holds the codes as exact bf16 with
// the fp32 scales beside them, and the softmax multiplies each score by its
// key's scale.
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
  static constexpr int QBA = (QB + 1023) / 1024 * 1024;  // one Q tile, 1 KB aligned
  static constexpr int OFF_Q = 0;                        // two Q tiles
  static constexpr int OFF_K = 2 * QBA;
  static constexpr int KBA = (KB + 1023) / 1024 * 1024;
  // K tiles per stage: 2 for quantised keys widened to hi + lo where a
  // 3-stage ring of them fits the 227 KB a CTA may hold (a 2-stage ring was
  // measured 40 % slower at r = 64), else 1 (bf16 keys, or exact bf16 codes
  // whose scales the softmax applies)
  static constexpr int KT = (KF != 0 && 2 * QBA + 3 * (2 * KBA + VB) + 2048 <= 227 * 1024) ? 2 : 1;
  static constexpr bool SCALE_IN_SOFTMAX = KF != 0 && KT == 1;
  static constexpr int SCB = SCALE_IN_SOFTMAX ? kBN * 4 : 0;  // a tile's key scales
  static constexpr int VOFF = KT * KBA;              // V tile offset in a stage
  static constexpr int STAGE = VOFF + VB;
  static constexpr int NST = (KT == 2 || 2 * QBA + 3 * (STAGE + SCB) + 2048 <= 200 * 1024) ? 3 : 2;
  static constexpr int OFF_SC = OFF_K + NST * STAGE;
  static constexpr int OFF_BAR = OFF_SC + NST * SCB;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;      // + slack to align the base to 1 KB
  static_assert(SMEM <= 227 * 1024, "shared memory");
  static constexpr uint32_t IDESC_S = instr_desc(kBM, kBN, false);
  static constexpr uint32_t IDESC_O = instr_desc(kBM, DV, true);
};

// Exact fp32 values of four int8 codes: each code, biased by 128, becomes the
// low byte of the float 2^23 + (c + 128), and 2^23 + 128 is subtracted.
__device__ __forceinline__ void i8x4_to_f32(uint32_t w, float2& a, float2& b) {
  const uint32_t x = w ^ 0x80808080u;
  uint32_t f0, f1, f2, f3;
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7540;" : "=r"(f0) : "r"(x));
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7541;" : "=r"(f1) : "r"(x));
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7542;" : "=r"(f2) : "r"(x));
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7543;" : "=r"(f3) : "r"(x));
  const float2 bias = make_float2(-8388736.0f, -8388736.0f);  // -(2^23 + 128)
  a = fadd2(make_float2(__uint_as_float(f0), __uint_as_float(f1)), bias);
  b = fadd2(make_float2(__uint_as_float(f2), __uint_as_float(f3)), bias);
}

// Exact fp32 values of eight int4 codes (element 2i in the low nibble of byte
// i, 2i+1 in its high nibble, 4-bit two's complement): c + 8 = nibble ^ 8
// becomes the low byte of 2^23 + (c + 8), and 2^23 + 8 is subtracted.
__device__ __forceinline__ void i4x8_to_f32(uint32_t w, float2 (&o)[4]) {
  const uint32_t t = w ^ 0x88888888u;
  const uint32_t lo = t & 0x0F0F0F0Fu, hi = (t >> 4) & 0x0F0F0F0Fu;
  const float2 bias = make_float2(-8388616.0f, -8388616.0f);  // -(2^23 + 8)
  uint32_t a[4], b[4];
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7540;" : "=r"(a[0]) : "r"(lo));
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7541;" : "=r"(a[1]) : "r"(lo));
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7542;" : "=r"(a[2]) : "r"(lo));
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7543;" : "=r"(a[3]) : "r"(lo));
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7540;" : "=r"(b[0]) : "r"(hi));
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7541;" : "=r"(b[1]) : "r"(hi));
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7542;" : "=r"(b[2]) : "r"(hi));
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7543;" : "=r"(b[3]) : "r"(hi));
#pragma unroll
  for (int i = 0; i < 4; ++i)
    o[i] = fadd2(make_float2(__uint_as_float(a[i]), __uint_as_float(b[i])), bias);
}

// x as two bf16 pairs with hi + lo = x to within 2^-17 |x|: hi = bf16(x), and
// x - hi (exact in fp32) rounded to bf16.  Low halves hold x.x.
__device__ __forceinline__ void split_bf16(float2 x, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(x.x, x.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  const float2 d = fadd2(x, make_float2(-__uint_as_float(hi << 16), -__uint_as_float(hi & 0xffff0000u)));
  const __nv_bfloat162 l = __floats2bfloat162_rn(d.x, d.y);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

struct Maps {
  CUtensorMap q, k, v;
  CUtensorMap klo;  // lo plane of widened quantised keys (two K tiles per stage)
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
__global__ void __launch_bounds__(kThreads, 1)
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
  uint64_t* c_full = o_full + 2;                // [NST] cached mode: the last tile landed
  uint64_t* sc_full = c_full + NST;             // [NST] key scales landed (scales in the softmax)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sc_full + NST);

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
      mbar_init(&k_full[s], 1);
      mbar_init(&v_full[s], 1);
      mbar_init(&kv_empty[s], 1);
      mbar_init(&c_full[s], 1);
      mbar_init(&sc_full[s], 1);
    }
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

  // In cached mode the tile holding the context's end is "relayed": it lands on
  // c_full, the TMA warp zeroes its value rows past the context (the cache may
  // hold anything there, and 0 * NaN would spread) and then publishes it on
  // k_full.  Other tiles go straight from the TMA to k_full.
  const bool relay = p.seq_lens != nullptr;
  auto relayed = [&](int j) { return relay && kv_len - j * kBN < kBN; };
  auto finish = [&](int j) -> bool {
    const int st = j % NST;
    unsigned char* sv = smem + C::OFF_K + st * C::STAGE + C::VOFF;
    const bool okc = mbar_wait(&c_full[st], 0, p.err) && mbar_wait(&v_full[st], (j / NST) & 1, p.err);
    if (!__all_sync(0xffffffffu, okc)) return false;
    const int first = max(kv_len - j * kBN, 0);
    const int per_box = (kBN - first) * 8;   // 16-byte pieces per value box
    for (int c = lane; c < per_box * C::V_NBOX; c += 32) {
      const int box = c / per_box, rem2 = c % per_box;
      *reinterpret_cast<uint4*>(sv + box * C::V_BOXB + (first + rem2 / 8) * 128 + (rem2 % 8) * 16) =
          make_uint4(0u, 0u, 0u, 0u);
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    __syncwarp();
    if (lane == 0) mbar_arrive(&k_full[st]);
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
        unsigned char* sv = sk + C::VOFF;
        uint64_t* kb = relayed(j) ? &c_full[st] : &k_full[st];
        if constexpr (KF == kKeyBF16) {
          mbar_arrive_expect_tx(kb, C::KB);
          for (int s2 = 0; s2 < nsub; ++s2)
            for (int i = 0; i < C::QK_NBOX; ++i)
              tma_load_3d(sk + i * C::QK_BOXB + s2 * bps * C::QK_SW, &maps.k, i * C::QK_BOX,
                          rows[s2], planes[s2], kb);
        } else {
          // widened keys from the workspace: [B*Hkv][kw_rows][r] planes, one box per tile
          mbar_arrive_expect_tx(kb, C::KT * C::KB);
          for (int i = 0; i < C::QK_NBOX; ++i) {
            tma_load_3d(sk + i * C::QK_BOXB, &maps.k, i * C::QK_BOX, j * kBN, kv_plane, kb);
            if constexpr (C::KT == 2)
              tma_load_3d(sk + C::KBA + i * C::QK_BOXB, &maps.klo, i * C::QK_BOX, j * kBN, kv_plane, kb);
          }
          if constexpr (C::SCALE_IN_SOFTMAX) {
            // the tile's key scales (rows past kw_rows are never weighted)
            const uint32_t bytes = static_cast<uint32_t>(min(kBN, p.kw_rows - j * kBN)) * 4u;
            mbar_arrive_expect_tx(&sc_full[st], bytes);
            bulk_g2s(smem + C::OFF_SC + st * C::SCB,
                     p.kw_scale + static_cast<size_t>(kv_plane) * p.kw_rows + j * kBN, bytes, &sc_full[st]);
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
    for (int j = 0; j < n_kv; ++j) {
      if (!issue(j)) break;
      if (relayed(j) && !finish(j)) break;
    }
  } else if (warp == 9) {
    // ------------------------------------------------------------------ MMA issuer
    {
      // descriptors of Q tile A and of the K / V tiles of stage 0; other
      // stages and K steps are start-address offsets from these
      const Desc dq = make_desc(smem_addr(smem + C::OFF_Q), 16, 8 * C::QK_SW, C::QK_LAYOUT);
      const Desc dk = make_desc(smem_addr(smem + C::OFF_K), 16, 8 * C::QK_SW, C::QK_LAYOUT);
      const Desc dv = make_desc(smem_addr(smem + C::OFF_K + C::VOFF), C::V_BOXB, 1024, 2u);
      auto issue_s = [&](int x, int st) {  // S_x = Q_x K^T
        const uint32_t qo = x * C::QBA, ko = st * C::STAGE;
#pragma unroll
        for (int k = 0; k < R / 16; ++k) {
          const uint32_t off = (k / C::KSTEP_PER_BOX) * C::QK_BOXB + (k % C::KSTEP_PER_BOX) * 32;
          mma_ss_e(tmem + x * 128, dq.at(qo + off), dk.at(ko + off), C::IDESC_S, k > 0);
        }
        if constexpr (C::KT == 2) {  // + Q_x lo^T
#pragma unroll
          for (int k = 0; k < R / 16; ++k) {
            const uint32_t off = (k / C::KSTEP_PER_BOX) * C::QK_BOXB + (k % C::KSTEP_PER_BOX) * 32;
            mma_ss_e(tmem + x * 128, dq.at(qo + off), dk.at(ko + C::KBA + off), C::IDESC_S, 1u);
          }
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
      if constexpr (C::SCALE_IN_SOFTMAX) {
        // quantised keys: the products are q . code; each key's fp32 scale turns
        // them into q . k (the scales arrive on sc_full)
        const int st = j % NST;
        if (!__all_sync(0xffffffffu, mbar_wait(&sc_full[st], (j / NST) & 1, p.err))) { ok = false; break; }
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
      static_assert(kParts == 2, "two key ranges of P");
      // pairs [i0, i1) of key range c into pk[i0 .. i1)
      auto compute = [&](int c, int i0, int i1, uint32_t* pk) {
#pragma unroll
        for (int i = i0; i < i1; ++i) {
          const int e = 2 * kPartPairs * c + 2 * i;
          const float2 t = ffma2(make_float2(__uint_as_float(v[e]), __uint_as_float(v[e + 1])),
                                 sl2x2, negm2);
          const float2 pr = make_float2(fast_exp2(t.x), fast_exp2(t.y));
          acc[i & 3] = fadd2(acc[i & 3], pr);
          __nv_bfloat162 b2 = __floats2bfloat162_rn(pr.x, pr.y);  // low half = column e
          pk[i] = *reinterpret_cast<uint32_t*>(&b2);
        }
      };
      auto publish = [&](int c) {
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(&p_full[kParts * x + c]);
      };
      uint32_t pk0[kPartPairs], pk1[kPartPairs];
      compute(0, 0, kPartPairs, pk0);
      tmem_st<kPartPairs>(tS + lane_off, pk0);
      if (j > 0 && __any_sync(0xffffffffu, resc)) {
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
      // the first half of range 1 while range 0's store lands, then range 0 is
      // published; same arithmetic and order of sums as range by range
      compute(1, 0, kPartPairs / 2, pk1);
      publish(0);
      compute(1, kPartPairs / 2, kPartPairs, pk1);
      tmem_st<kPartPairs>(tS + lane_off + kPartPairs, pk1);
      publish(1);
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
      // the whole O row with one TMEM wait (the score registers are free by now)
      uint32_t o[DV];
      if constexpr (DV == 128) tmem_ld128(tO + lane_off, o);
      else tmem_ld64(tO + lane_off, o);
#pragma unroll
      for (int c = 0; c < DV / 32; ++c) {
        const uint32_t* v = o + 32 * c;
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

// Widens the keys of each sequence's context, tokens 0 .. seq_lens[b] + S - 1
// of an int8 / int4 cache (contiguous or paged), into the workspace planes
// [B*Hkv][kw_rows][r] that the prefill loads by TMA: hi and lo of
// scale * code (KT = 2), or the codes as exact bf16 with the fp32 scales in
// sc[B*Hkv][kw_rows] (KT = 1).  Once per token, where widening inside the
// prefill would redo it for every query tile pair that reads the tile.  One
// thread per 8 elements of one token; rows past a context are left as they
// are (their scores are masked and their value rows zeroed).
template <int R, int KF, int KT>
__global__ void __launch_bounds__(256) key_widen_kernel(const PrefillParams p, __nv_bfloat16* hi,
                                                        __nv_bfloat16* lo, float* sc) {
  constexpr int PPR = R / 8;
  const long long i = static_cast<long long>(blockIdx.x) * 256 + threadIdx.x;
  if (i >= static_cast<long long>(p.B) * p.Hkv * p.kw_rows * PPR) return;
  const int piece = static_cast<int>(i % PPR);
  const long long tok = i / PPR;
  const int t = static_cast<int>(tok % p.kw_rows);
  const int plane = static_cast<int>(tok / p.kw_rows);  // b * Hkv + g
  const int b = plane / p.Hkv, g = plane - b * p.Hkv;
  // seq_lens[b] clamped as the prefill kernel clamps it (and records the error)
  const int L0 = min(max(p.seq_lens[b], 0), p.kv_limit - p.S);
  if (t >= L0 + p.S) return;
  long long row;  // cache row of token t
  if (p.page_size == 0) {
    row = static_cast<long long>(plane) * p.capacity + t;
  } else {
    int page = p.page_table[static_cast<long long>(b) * p.max_pages + (t >> p.page_shift)];
    if (page < 0 || page >= p.num_pages) {
      record_error(p.err, TK_DEVERR_INDEX);
      page = 0;
    }
    row = (static_cast<long long>(page) * p.Hkv + g) * p.page_size + (t & (p.page_size - 1));
  }
  const float s = p.k_scale[row];
  const size_t o = static_cast<size_t>(tok) * R + piece * 8;
  if constexpr (KT == 2) {
    float2 x[4];
    if constexpr (KF == kKeyInt8) {
      const uint2 w = *reinterpret_cast<const uint2*>(static_cast<const int8_t*>(p.k) + row * R + piece * 8);
      i8x4_to_f32(w.x, x[0], x[1]);
      i8x4_to_f32(w.y, x[2], x[3]);
    } else {
      i4x8_to_f32(*reinterpret_cast<const uint32_t*>(static_cast<const uint8_t*>(p.k) + row * (R / 2) +
                                                     piece * 4),
                  x);
    }
    const float2 s2 = make_float2(s, s);
    uint4 h, l;
    split_bf16(fmul2(x[0], s2), h.x, l.x);
    split_bf16(fmul2(x[1], s2), h.y, l.y);
    split_bf16(fmul2(x[2], s2), h.z, l.z);
    split_bf16(fmul2(x[3], s2), h.w, l.w);
    *reinterpret_cast<uint4*>(hi + o) = h;
    *reinterpret_cast<uint4*>(lo + o) = l;
  } else {
    uint4 h;
    if constexpr (KF == kKeyInt8) {
      const uint2 w = *reinterpret_cast<const uint2*>(static_cast<const int8_t*>(p.k) + row * R + piece * 8);
      i8x4_to_bf16(w.x, h.x, h.y);
      i8x4_to_bf16(w.y, h.z, h.w);
    } else {
      i4x8_to_bf16(*reinterpret_cast<const uint32_t*>(static_cast<const uint8_t*>(p.k) + row * (R / 2) +
                                                      piece * 4),
                   h.x, h.y, h.z, h.w);
    }
    *reinterpret_cast<uint4*>(hi + o) = h;
    if (piece == 0) sc[tok] = s;
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
  PrefillParams pp = p;
  bool ok = make_map(&maps.q, p.q, R, p.S, p.B * p.Hq, C::QK_BOX, kBM, C::QK_SW) &&
            make_map(&maps.v, p.v, DV, kv_rows, kv_planes, 64, box_rows, 128);
  __nv_bfloat16 *hi = nullptr, *lo = nullptr;
  float* sc = nullptr;
  if constexpr (KF == kKeyBF16) {
    ok = ok && make_map(&maps.k, p.k, R, kv_rows, kv_planes, C::QK_BOX, box_rows, C::QK_SW);
  } else {
    // workspace: plane 0 = hi (or the bf16 codes), then lo (or the scales)
    if (!p.kw || p.kw_bytes < prefill_workspace_bytes(p.B, p.Hkv, R, DV, KF, p.kw_rows) ||
        p.kw_rows % 4 != 0 || p.kw_rows < p.kv_limit)
      return cudaErrorInvalidValue;
    const size_t plane = static_cast<size_t>(p.B) * p.Hkv * p.kw_rows * R;
    hi = static_cast<__nv_bfloat16*>(p.kw);
    if constexpr (C::KT == 2) lo = hi + plane;
    else sc = reinterpret_cast<float*>(hi + plane);
    pp.kw_scale = sc;
    ok = ok && make_map(&maps.k, hi, R, p.kw_rows, p.B * p.Hkv, C::QK_BOX, kBN, C::QK_SW);
    if constexpr (C::KT == 2)
      ok = ok && make_map(&maps.klo, lo, R, p.kw_rows, p.B * p.Hkv, C::QK_BOX, kBN, C::QK_SW);
  }
  if (!ok) return cudaErrorInvalidValue;
  auto kern = prefill_kernel<R, DV, KF>;
  const int smem = C::SMEM;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const long n_qt = (p.S + kBM - 1) / kBM;
  const long grid = (n_qt + 1) / 2 * p.B * p.Hq;  // one CTA per query tile pair
  if (grid > 0x7fffffffL) return cudaErrorInvalidConfiguration;
  if constexpr (KF != kKeyBF16) {
    const long long n = static_cast<long long>(p.B) * p.Hkv * p.kw_rows * (R / 8);
    key_widen_kernel<R, KF, C::KT><<<static_cast<unsigned>((n + 255) / 256), 256, 0, stream>>>(p, hi, lo, sc);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  // about 48 MB of K/V per head group
  const long head_bytes = static_cast<long>(p.seq_lens ? p.kv_limit : p.S) * (R + DV) * 2;
  pp.head_group = static_cast<int>(std::max(1L, std::min<long>(p.B * p.Hq, (48L << 20) / head_bytes)));
  kern<<<static_cast<unsigned>(grid), kThreads, smem, stream>>>(maps, pp);
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

template <int R, int DV>
size_t ws_bytes_t(int B, int Hkv, int k_fmt, int rows) {
  const size_t plane = static_cast<size_t>(B) * Hkv * rows * R * 2;  // bf16 [B*Hkv][rows][r]
  bool two = PCfg<R, DV, kKeyInt8>::KT == 2;
  if constexpr (R >= 32) {
    if (k_fmt == kKeyInt4) two = PCfg<R, DV, kKeyInt4>::KT == 2;
  } else {
    if (k_fmt == kKeyInt4) return 0;  // int4 keys need r >= 32
  }
  return two ? 2 * plane : plane + static_cast<size_t>(B) * Hkv * rows * 4;
}

size_t prefill_workspace_bytes(int B, int Hkv, int R, int DV, int k_fmt, int rows) {
  if (k_fmt == kKeyBF16 || B <= 0 || Hkv <= 0 || rows <= 0 || (DV != 64 && DV != 128)) return 0;
  switch (R) {
    case 16: return DV == 64 ? ws_bytes_t<16, 64>(B, Hkv, k_fmt, rows) : ws_bytes_t<16, 128>(B, Hkv, k_fmt, rows);
    case 32: return DV == 64 ? ws_bytes_t<32, 64>(B, Hkv, k_fmt, rows) : ws_bytes_t<32, 128>(B, Hkv, k_fmt, rows);
    case 64: return DV == 64 ? ws_bytes_t<64, 64>(B, Hkv, k_fmt, rows) : ws_bytes_t<64, 128>(B, Hkv, k_fmt, rows);
    case 128: return DV == 64 ? ws_bytes_t<128, 64>(B, Hkv, k_fmt, rows) : ws_bytes_t<128, 128>(B, Hkv, k_fmt, rows);
  }
  return 0;
}

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
