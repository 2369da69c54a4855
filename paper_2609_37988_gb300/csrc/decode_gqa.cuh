// decode_gqa.cuh -- split-K decode attention over one GQA anchor (sm_103a).
//
// Computes, for every query head h of sequence b (Sec. 2.1 GQA; the depth
// axis only changes which anchor is read):
//     out[b,h] = sum_t softmax_t(sigma <q[b,h], k_t>) v_t ,  k_t/v_t of KV head h/G
// over the positions of b (or its kept list, Sec. 3.4), with k_t and v_t
// dequantised on the fly (grouped asymmetric codes, Appendix C.3).
//
// Grid (split, kv head, batch); 4 warps per CTA; each CTA streams its
// context split in tiles of 64 positions through a cp.async ring of NST
// shared-memory stages (16-byte copies; an eviction list turns the same
// copies into a gather).  Warp w owns tile rows [16w, 16w+16) and keeps its
// own online-softmax state; the four states merge in shared memory at the
// end and either write the output (one split) or a split-K partial.
//
// Both products run on the tensor cores with mma.m16n8k16 (fp32 accumulate):
//   scores  S^T[16 pos x 8 heads] = K[16 x 16 ch] * Q^T, the G <= 8 query
//           heads of the KV head share one read of every key byte;
//   values  O^T[16 ch x 8 heads] += V^T[16 ch x 16 pos] * P^T.
// Codes enter the MMA as exact f16 subnormals (the bit pattern c is the
// half c * 2^-24; the factor 2^-24 is undone on the fp32 side).  Scale and
// zero stay fp32 and are applied outside the MMA, so quantised operands lose
// nothing:
//   keys, per-token groups:   s_t = sum_g sc_tg D_tg + z_tg Qs_g
//   keys, per-channel groups: scale folded into the query per group of
//                             positions, zero term  sum_i q_i z_Gi
//   values: P'_g = p * sc_tg per channel group (hi/lo f16 split), plus
//           sum_t p_t z_tg added once at the end.
// bf16 caches multiply bf16 operands directly; P is split into hi + lo
// bf16 halves so the value product keeps ~16 significant bits.
// The symmetric per-vector scheme (KAX == kKaxSym; the paper's quantiser,
// Appendix C.3) is the per-token case with one group per row: codes stored
// as u = code + q, so x = s u - q s, i.e. scale s and zero -q s, with the
// bf16 scales streamed from the anchor's scale plane beside the records.
// 2-bit codes (this scheme only) enter the MMA like 4-bit ones, as masked
// fields of a word at weights 4^e that the query (keys) or the final
// accumulator scale (values) undoes.
#pragma once
#include <cuda.h>  // CUtensorMap (the gather's row copies)
#include <math.h>
#include <string.h>

#include "common.cuh"
#include "kernels.h"
#include "layout.h"

namespace kvk {

// key-axis template value of the symmetric per-vector scheme
constexpr int kKaxSym = 2;

template <int BITS, int D, int KAX, int GS>
struct GqaCfg {
  static constexpr bool BF = (BITS == 16);
  static constexpr bool QUANT = !BF;
  static constexpr bool SYM = QUANT && KAX == kKaxSym;  // scales in the scale plane
  static constexpr bool KPT = QUANT && (KAX == 0 || SYM);  // per-token key groups
  static constexpr bool KPC = QUANT && KAX == 1;  // per-channel key groups
  static constexpr int KS = D / 16;               // k-steps (= value M-blocks)
  static constexpr int NG = QUANT ? D / GS : 1;   // channel groups per row
  static constexpr int KB = D * BITS / 8;         // K (and V) section bytes
  static constexpr int MB = (QUANT && !SYM) ? ((NG * 8 + 15) & ~15) : 0;
  static constexpr int REC = 2 * KB + (KPT ? MB : 0) + (QUANT ? MB : 0);
  static constexpr int CPR = REC / 16;            // 16-byte chunks per record
  static constexpr int SK = KB / 4;               // bytes of one lane's K segment
  static constexpr int NWK = SK / 4;              // words of one lane's K segment
  static constexpr int SV = KB / 8;               // bytes of one lane's V segment
  static constexpr int NWV = SV / 4;
  // shared-memory planes of one stage (row = tile position)
  static constexpr int KSTR = KB;
  static constexpr bool KSWZ = KB >= 128;
  static constexpr int VSTR = KB >= 128 ? KB : (KB == 64 ? 80 : 48);
  static constexpr int VSWZ = KB >= 256 ? 2 : (KB == 128 ? 1 : 0);
  static constexpr int KP_OFF = 0;
  static constexpr int VP_OFF = KP_OFF + kTile * KSTR;
  static constexpr int KM_OFF = VP_OFF + kTile * VSTR;
  static constexpr int VM_OFF = KM_OFF + (KPT ? kTile * MB : 0);
  static constexpr int KG_OFF = VM_OFF + (QUANT ? kTile * MB : 0);
  // row blocks of 16 per warp and tile height: two blocks for per-token
  // 4-bit keys (more independent work per warp, shared softmax reductions)
  static constexpr int RB = (KPT && BITS <= 4) ? 2 : 1;
  static constexpr int TILE = 64 * RB;
  static constexpr int KG_ROWS = KPC ? kTile / GS : 0;
  static constexpr int NCH = REC / 16;            // 16-byte chunks per record
  static constexpr float QL = SYM ? (float)((1 << (BITS - 1)) - 1) : 0.f;  // symmetric q
  // Quantised caches: a stage is 64 raw records (one bulk copy) followed by
  // the tile's key-group metadata rows.  bf16 caches: planes filled by
  // 16-byte copies with conflict-free swizzles.
  static constexpr bool TMA = QUANT;
  static constexpr int KG_OFF_T = TILE * REC;
  static constexpr int SC_OFF_T = TILE * REC;     // symmetric: one scale word per row
  static constexpr int STAGE = TMA ? KG_OFF_T + KG_ROWS * D * 8 + (SYM ? TILE * 4 : 0)
                                   : KG_OFF + KG_ROWS * D * 8;
  static constexpr int QSTR = D + 4;  // padded query row (floats): conflict-free head rows
  // padded to 128 bytes: stages (tensor-map copy destinations) start 128-byte aligned
  static constexpr int Q_BYTES = (8 * QSTR * 4 + 2 * 8 * NG * 4 + 127) & ~127;
  // per-channel keys: the query folded with each group's scales, once per
  // tile, in the score MMA's fragment order ([KG_ROWS][KS][32] x 16 bytes),
  // and the zero-point terms per warp ([4][KG_ROWS][8] floats)
  static constexpr int FOLD_BYTES = KPC ? KG_ROWS * KS * 32 * 16 : 0;
  static constexpr int ZRED_BYTES = KPC ? 4 * KG_ROWS * 8 * 4 : 0;
  // stages: bf16 planes three (head_dim 128: two CTAs per SM, ~190 KB of
  // copies in flight per SM, the decode bound by HBM); quantised stages
  // four where they and the rest fit four CTAs per SM (57 KB each), else
  // three or two by stage size
  static constexpr int FIXED = Q_BYTES + FOLD_BYTES + ZRED_BYTES + 24 * 4;
  static constexpr int NST = !TMA ? 3
                             : KPC ? (FIXED + 4 * STAGE <= 57344 ? 4 : (FIXED + 3 * STAGE <= 57344 ? 3 : (STAGE <= 20480 ? 3 : 2)))
                                   : (STAGE <= 13312 ? 4 : (STAGE <= 20480 ? 3 : 2));
  static_assert(TMA || RB == 1, "plane layout holds 64-row tiles");
  static constexpr int BAR_OFF = Q_BYTES + NST * STAGE;
  static constexpr int GMASK_OFF = BAR_OFF + (TMA ? 16 * NST : 0);  // two mbarrier sets
  // The kept-list gather of grouped per-token records copies whole records
  // with tensor-map row copies (four rows per instruction): the records land
  // as stored, so the consumer reads each row's value-chunk rotation (one
  // byte per row and stage) instead of deriving it from the row.
  static constexpr bool GTMA = QUANT && !SYM && KPT;
  static constexpr int ROT_OFF = GMASK_OFF + (TMA ? 16 * NST : 0);
  static constexpr int FOLD_OFF = (ROT_OFF + (GTMA ? NST * TILE : 0) + 15) & ~15;  // 16-byte stores
  static constexpr int SMEM = FOLD_OFF + FOLD_BYTES + ZRED_BYTES;
  // CTAs per SM the register budget is sized for: four where four fit in
  // shared memory (228 KB per SM, 1 KB reserved per CTA), else three
  static constexpr int MIN_CTAS = (!BF && 4 * (SMEM + 1024) <= 233472) ? 4 : 3;
  static_assert(REC % 16 == 0, "records are 16-byte multiples");
  static_assert(Q_BYTES % 16 == 0 && STAGE % 16 == 0 && FOLD_OFF % 16 == 0, "16-byte aligned regions");
  static_assert(!GTMA || (Q_BYTES % 128 == 0 && STAGE % 128 == 0 && (4 * REC) % 128 == 0),
                "row-copy destinations 128-byte aligned");
  static_assert(BITS != 2 || SYM, "2-bit codes exist for the symmetric scheme only");
  static_assert(!SYM || (D == 128 && GS == D), "symmetric rows are 128 channels, one group");
  static_assert(!QUANT || (GS % 16 == 0 && D % GS == 0), "groups are whole k-steps");
  static_assert(4 * 8 * (D + 2) * 4 <= NST * STAGE, "merge scratch fits the stages");
};

__device__ __forceinline__ int kswz(bool on, int t, int u) { return on ? (u ^ ((t & 1) << 2)) : u; }
__device__ __forceinline__ int vswz(int mode, int t, int u) {
  if (mode == 1) return u ^ (t & 6);
  if (mode == 2) return u ^ (((t >> 1) & 1) | (((t >> 2) & 1) << 2));
  return u;
}

// Tensor-map row copy of four records: rows r0..r3 of the anchor's record
// table (one box = one record) land back to back at dst, completing on bar.
__device__ __forceinline__ void tma_rows4(void *dst, const CUtensorMap *map, int r0, int r1, int r2,
                                          int r3, uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile::gather4.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(r0), "r"(r1), "r"(r2), "r"(r3),
      "r"(smem_u32(bar))
      : "memory");
}

// Codes as f16 operands: a code c placed in the low bits of a zero f16 bit
// pattern is the subnormal c * 2^-24, exact, and the tensor cores multiply
// it exactly into fp32.  Every code-side product therefore carries a factor
// 2^-24, undone once on the fp32 side (kCodeScale).
constexpr float kCodeUnit = 5.9604644775390625e-8f;  // 2^-24
constexpr float kCodeScale = 16777216.f;            // 2^24
// f16 pair (c_lo, c_hi) * 2^-24 from two bytes picked by `sel` (PRMT; the
// selector's other nibbles pick zero bytes).
__device__ __forceinline__ uint32_t u8pair_f16(uint32_t x, uint32_t sel) {
  return __byte_perm(x, 0u, sel);
}
// f16 pair of the nibbles under `mask` (low nibble: c * 2^-24, high nibble:
// 16 c * 2^-24).
__device__ __forceinline__ uint32_t nib_f16(uint32_t x, uint32_t mask) { return x & mask; }

// The key code of channel ch enters the score MMA at weight 4^e (the query
// fragment of that channel carries 4^-e): 4-bit codes in a high nibble
// (slots 8..15 of a k-step) e = 2; 2-bit codes e = 2 (k-step mod 2) +
// (slot >= 8); else e = 0.  key_weight(ch, s) = 4^(s e), s = +1 or -1,
// built from its exponent bits (exact, no division).
template <int BITS>
__device__ __forceinline__ int key_weight_exp(int ch) {
  if constexpr (BITS == 4) return ((ch & 15) >= 8) ? 2 : 0;
  if constexpr (BITS == 2) return 2 * ((ch >> 4) & 1) + ((ch & 15) >= 8);
  return 0;
}
template <int BITS>
__device__ __forceinline__ float key_weight(int ch, int sgn) {
  return __int_as_float((127 + 2 * sgn * key_weight_exp<BITS>(ch)) << 23);
}

// The decode of one unit (sequence b, KV head kvh) over items [i0, i1) of
// its positions or kept list (i1 < 0: to the end), written to partial slot
// `slot`, or normalised to the output when a.out is set.  The copy ring
// starts at tile 0 on mbarrier set `bset` (NST fresh mbarriers, initialised
// by the caller; a CTA decoding two units uses one set for each, so that
// both run the same code with stage and phase fixed by the tile number).
// rows: the anchor's record table as a tensor map (kept-list gather of
// grouped per-token records).  Returns false when a bounded wait gave up.
// GATHER: the rows come from the anchor's kept-position list (compiled
// separately so that the contiguous path carries none of its state).
template <int BITS, int D, int KAX, int GS, bool GATHER>
__device__ __forceinline__ bool gqa_decode_unit(const GqaDecodeArgs &a, const CUtensorMap *rows,
                                                const int b, const int kvh, const int i0,
                                                const int i1_req, const int slot, const int bset) {
  using C = GqaCfg<BITS, D, KAX, GS>;
  constexpr bool BF = C::BF;
  constexpr int KS = C::KS, NG = C::NG;
  extern __shared__ __align__(128) uint8_t smem[];
  constexpr int QSTR = C::QSTR;
  float *q_s = reinterpret_cast<float *>(smem);        // [8][QSTR]
  float *qs_s = q_s + 8 * QSTR;                        // [8][NG] query sums per group
  uint8_t *stages = smem + C::Q_BYTES;

  const GqaView &v = a.v;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, c = lane & 3;
  const int len = v.lens[b];
  // kept-position lists exist only with per-token key metadata or bf16
  // caches (rejected by the host for per-channel keys)
  constexpr bool gather = GATHER && !C::KPC;
  const int kunit = v.kept_per_head ? b * v.Hkv + kvh : b;  // whose kept list
  const int n_items = gather ? min(v.kept_n[kunit], v.kept_cap) : len;
  const int i1 = i1_req < 0 ? n_items : min(i1_req, n_items);
  const int Tq = C::KPC ? (len / GS) * GS : len;  // positions held as codes
  const bool use_lo = a.q_f32 != 0;
  const int32_t *kept = v.kept_idx + (size_t)kunit * v.kept_cap;

  // The copy producer comes first, so the first tiles are in flight while
  // the query set-up below runs.
  const size_t slab = (size_t)b * v.Hkv + kvh;
  const uint8_t *rec = v.rec + slab * (size_t)v.cap * C::REC;
  const float2 *gmeta = C::KPC ? v.gmeta + slab * (size_t)(v.cap / GS) * D : nullptr;
  const uint32_t *scl = C::SYM ? v.scales + slab * (size_t)v.cap : nullptr;
  const int n_tiles = i1 > i0 ? (i1 - i0 + C::TILE - 1) / C::TILE : 0;

  // ---- producer: one tile of records into one stage ----------------------
  // Thread tid copies chunk columns u = tid/8 + 16j of rows tid%8 + 8k.  All
  // shared-memory swizzles depend on the row only through row % 8, so each
  // (thread, column) has one destination offset and one plane stride, and a
  // chunk costs two adds, a compare and the copy.
  constexpr int NCOL = (C::CPR + 15) / 16;
  const int crow = tid & 7, ccol = tid >> 3;
  int cdst0[NCOL], cstr[NCOL];
#pragma unroll
  for (int j = 0; j < NCOL; ++j) {
    const int u = ccol + 16 * j;
    const int ub = 16 * u;
    int off, str;
    if (ub < C::KB) {
      off = C::KP_OFF + crow * C::KSTR + 16 * kswz(C::KSWZ, crow, u);
      str = C::KSTR;
    } else if (ub < 2 * C::KB) {
      off = C::VP_OFF + crow * C::VSTR + 16 * vswz(C::VSWZ, crow, u - C::KB / 16);
      str = C::VSTR;
    } else if (C::KPT && ub < 2 * C::KB + C::MB) {
      off = C::KM_OFF + crow * C::MB + (ub - 2 * C::KB);
      str = C::MB;
    } else {
      off = C::VM_OFF + crow * C::MB + (ub - 2 * C::KB - (C::KPT ? C::MB : 0));
      str = C::MB;
    }
    cdst0[j] = (u < C::CPR) ? off : -1;
    cstr[j] = 8 * str;
  }
  auto issue_cp = [&](int t, int s) {
    const int base = i0 + t * kTile;
    uint8_t *st = stages + s * C::STAGE;
#pragma unroll
    for (int k = 0; k < kTile / 8; ++k) {
      const int item = base + crow + 8 * k;
      bool valid = item < i1;
      int pos = item;
      if (gather && valid) {
        pos = kept[item];
        if (pos < 0 || pos >= len) {
          valid = false;
          if (ccol == 0) set_err(a.err, 1);
        }
      }
      const uint8_t *src = rec + (size_t)(valid ? pos : 0) * C::REC + 16 * ccol;
#pragma unroll
      for (int j = 0; j < NCOL; ++j)
        if (cdst0[j] >= 0) cp_async16(st + cdst0[j] + k * cstr[j], src + 256 * j, valid);
    }
    if constexpr (C::KPC) {
      const int g0 = base / GS;
      constexpr int CPRow = D * 8 / 16;
      for (int q = tid; q < C::KG_ROWS * CPRow; q += 128) {
        const int row = q / CPRow, u = q - row * CPRow;
        const int G = g0 + row;
        const bool valid = (G + 1) * GS <= len;
        const uint8_t *src =
            reinterpret_cast<const uint8_t *>(gmeta + (size_t)(valid ? G : 0) * D) + 16 * u;
        cp_async16(st + C::KG_OFF + row * D * 8 + 16 * u, src, valid);
      }
    }
  };

  // bulk-copy producer (quantised caches): one copy per tile, or one per
  // kept record; rows that get no copy are zero-filled so stale bytes never
  // reach the arithmetic.
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + C::BAR_OFF) + bset * C::NST;
  // gather: kept position of row (TILE/4) warp + lane of the next tile to
  // issue, and per stage one row-validity word per warp
  uint32_t *gmask = reinterpret_cast<uint32_t *>(smem + C::GMASK_OFF);
  uint8_t *rotb = smem + C::ROT_OFF;  // [stage][row] value-chunk rotation (row gather)
  int gidx_next = -1;
  if constexpr (C::TMA) {
    if (gather) {
      const int r = i0 + (C::TILE / 4) * warp + lane;
      gidx_next = (lane < C::TILE / 4 && r < i1) ? kept[r] : -1;
    }
  }
  auto zero_rows = [&](uint8_t *st, int r_lo, int r_hi) {  // rows [r_lo, r_hi), all threads
    uint4 *p = reinterpret_cast<uint4 *>(st + r_lo * C::REC);
    const int n = (r_hi - r_lo) * (C::REC / 16);
    for (int q = tid; q < n; q += 128) p[q] = make_uint4(0, 0, 0, 0);
  };
  auto issue_tma = [&](int t, int s) {
    const int base = i0 + t * C::TILE;
    uint8_t *st = stages + s * C::STAGE;
    const int nrows = min(C::TILE, i1 - base);
    int kgv = 0;  // complete key groups of this tile (per-channel keys)
    if constexpr (C::KPC) kgv = max(0, min(C::KG_ROWS, len / GS - base / GS));
    if (!gather) {
      if (tid == 0) {
        // symmetric scales: whole 16-byte groups of 4 words (the slab's
        // capacity is a multiple of 64 positions, so they stay inside it)
        const int scb = C::SYM ? ((nrows + 3) & ~3) * 4 : 0;
        fence_proxy_async();
        mbar_expect_tx(&bars[s], nrows * C::REC + kgv * D * 8 + scb);
        bulk_g2s(st, rec + (size_t)base * C::REC, nrows * C::REC, &bars[s]);
        if (C::KPC && kgv > 0)
          bulk_g2s(st + C::KG_OFF_T, gmeta + (size_t)(base / GS) * D, kgv * D * 8, &bars[s]);
        if (C::SYM) bulk_g2s(st + C::SC_OFF_T, scl + base, scb, &bars[s]);
      }
      if (nrows < C::TILE) zero_rows(st, nrows, C::TILE);
    } else {
      // gather: warp w copies rows [RPW w, RPW (w+1)) of the tile with
      // 16-byte copies.  Lane l holds the kept position of row RPW w + l,
      // loaded one tile ahead (gidx_next) so that its latency hides behind
      // the current tile's arithmetic; the warp's row-validity bits go to
      // the stage's mask words, read by the consumer instead of the list.
      // Rows without a valid kept position are zero-filled by the copy.
      constexpr int CPRR = C::REC / 16;  // 16-byte chunks per record
      constexpr int RPW = C::TILE / 4;   // rows per warp (<= 32)
      const int myidx = gidx_next;
      {
        const int nrow = base + C::TILE + RPW * warp + lane;  // same row, next tile
        gidx_next = (lane < RPW && nrow < i1) ? kept[nrow] : -1;
      }
      bool mine = lane < RPW && RPW * warp + lane < nrows;
      if (mine && (myidx < 0 || myidx >= len)) {
        mine = false;
        set_err(a.err, 1);
      }
      const uint32_t vm = __ballot_sync(0xffffffffu, mine);
      if (lane == 0) gmask[s * 4 + warp] = vm;
      if constexpr (C::GTMA) {
        // whole records by tensor-map row copies, four rows per copy: lane j
        // < RPW / 4 copies the warp's rows 4j .. 4j + 3.  A row without a
        // valid position copies the slab's position 0 instead (a real
        // record: the consumer masks the row and zeroes its value scales).
        // Each row's value-chunk rotation goes to the stage's rotation bytes.
        const int trow = (int)(slab * (size_t)v.cap) + (mine ? myidx : 0);
        if (lane < RPW)
          rotb[s * C::TILE + RPW * warp + lane] = (uint8_t)(mine ? v_rot(myidx, C::REC, C::KB / 16) : 0);
        const int q = 4 * (lane & 7);
        const int r0 = __shfl_sync(0xffffffffu, trow, q), r1 = __shfl_sync(0xffffffffu, trow, q + 1);
        const int r2 = __shfl_sync(0xffffffffu, trow, q + 2), r3 = __shfl_sync(0xffffffffu, trow, q + 3);
        if (tid == 0) mbar_expect_tx(&bars[s], C::TILE * C::REC);
        if (lane < RPW / 4) {
          fence_proxy_async();
          tma_rows4(st + (RPW * warp + 4 * lane) * C::REC, rows, r0, r1, r2, r3, &bars[s]);
        }
        return;
      }
      // value chunks (grouped) or whole records (symmetric) are stored
      // rotated by the position and read rotated by the shared-memory row:
      // chunk u of the record moves accordingly
      constexpr int VC0 = C::KB / 16, NC = C::KB / 16;
      uint8_t *wst = st + RPW * warp * C::REC;
#pragma unroll 3
      for (int q0 = 0; q0 < RPW * CPRR; q0 += 32) {
        const int q = q0 + lane, j = q / CPRR, u = q - j * CPRR;
        const int pos = __shfl_sync(0xffffffffu, myidx, j & 31);
        if (q < RPW * CPRR) {
          const bool valid = (vm >> (j & 31)) & 1u;
          int ud = u;
          if constexpr (C::SYM)
            ud = (u - sym_rot(pos, C::NCH) + sym_rot(RPW * warp + j, C::NCH)) & (C::NCH - 1);
          else if (u >= VC0 && u < VC0 + NC)
            ud = VC0 + ((u - VC0 - v_rot(pos, C::REC, NC) + v_rot(RPW * warp + j, C::REC, NC)) &
                        (NC - 1));
          cp_async16(wst + j * C::REC + 16 * ud, rec + (size_t)(valid ? pos : 0) * C::REC + 16 * u,
                     valid);
        }
      }
      if constexpr (C::SYM) {
        if (lane < RPW)
          cp_async4(st + C::SC_OFF_T + 4 * (RPW * warp + lane), scl + (mine ? myidx : 0), mine);
      }
    }
  };
  auto issue = [&](int t, int s) {
    if constexpr (C::TMA)
      issue_tma(t, s);
    else
      issue_cp(t, s);
  };

  // completion by cp.async groups (bf16 planes, the chunked gather) or by
  // the stages' mbarriers (bulk and tensor-map row copies)
  const bool use_cp = !C::TMA || (gather && !C::GTMA);
#pragma unroll
  for (int s = 0; s < C::NST - 1; ++s) {
    if (s < n_tiles) issue(s, s);
    if (use_cp) cp_async_commit();
  }

  // the query rows: eight consecutive channels per thread, read with 16-byte
  // loads issued together (one memory round trip); heads past G are zero
  if (tid * 8 < 8 * D) {
    const int h = (tid * 8) / D, ch = (tid * 8) % D;
    float x[8];
    if (h < a.G) {
      const size_t qi = ((size_t)b * a.Hq + (size_t)kvh * a.G + h) * D + ch;
      if (a.q_f32) {
        const float4 *qp = reinterpret_cast<const float4 *>(static_cast<const float *>(a.q) + qi);
        const float4 x0 = qp[0], x1 = qp[1];
        x[0] = x0.x; x[1] = x0.y; x[2] = x0.z; x[3] = x0.w;
        x[4] = x1.x; x[5] = x1.y; x[6] = x1.z; x[7] = x1.w;
      } else {
        const uint4 w = *reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(a.q) + qi);
        const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          x[2 * i] = __uint_as_float(ws[i] << 16);
          x[2 * i + 1] = __uint_as_float(ws[i] & 0xffff0000u);
        }
      }
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) x[i] = 0.f;
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) q_s[h * QSTR + ch + i] = x[i];
  }
  __syncthreads();
  // per-token key groups: query sums Qs of every (head, channel group), of
  // the f16 values the score MMA actually uses, times 2^-24 like the code
  // products; 128 / (8 NG) lanes per (head, group), reduced with shuffles.
  if constexpr (C::KPT) {
    constexpr int ITEMS = 8 * NG, LPI = 128 / ITEMS, CPL = GS / LPI;
    const int item = tid / LPI, sub = tid % LPI;
    const int h = item / NG, gi = item % NG;
    const bool use_lo0 = a.q_f32 != 0;
    float sq = 0.f;
#pragma unroll 4
    for (int k = 0; k < CPL; ++k) {
      const int ch = gi * GS + sub * CPL + k;
      const float w = key_weight<BITS>(ch, 1);  // a power of two: exact scaling
      const float x = q_s[h * QSTR + ch];
      const float xs = x * key_weight<BITS>(ch, -1);
      float xe = __half2float(__float2half_rn(xs));
      if (use_lo0) xe += __half2float(__float2half_rn(xs - xe));
      sq += w * xe;
    }
#pragma unroll
    for (int off = 1; off < LPI; off <<= 1) sq += __shfl_xor_sync(0xffffffffu, sq, off);
    if (sub == 0) qs_s[item] = sq * kCodeUnit;
    __syncthreads();
  }

  // ---- query fragments (B operand of the score MMA), head n = g ----------
  // Built once per CTA by warp 0 and kept in shared memory over the query
  // rows (dead from here on): per k-step js, the 32 lanes' hi pairs at
  // qf[64 js + lane] and lo pairs at qf[64 js + 32 + lane].
  uint2 *qf = reinterpret_cast<uint2 *>(q_s);
  if constexpr (!C::KPC) {
    static_assert(KS * 64 * 8 <= 8 * QSTR * 4, "query fragments fit the query rows");
    uint32_t hb[KS][2], lb[KS][2];
    if (warp == 0) {
#pragma unroll
      for (int js = 0; js < KS; ++js) {
        const float *qh = q_s + g * QSTR + 16 * js;
        // inverse code weights of this lane's channels (powers of two)
        const float w0 = key_weight<BITS>(16 * js, -1), w1 = key_weight<BITS>(16 * js + 8, -1);
        split2<BF>(qh[2 * c] * w0, qh[2 * c + 1] * w0, hb[js][0], lb[js][0]);
        split2<BF>(qh[2 * c + 8] * w1, qh[2 * c + 9] * w1, hb[js][1], lb[js][1]);
      }
    }
    __syncthreads();  // every read of the query rows is done
    if (warp == 0) {
#pragma unroll
      for (int js = 0; js < KS; ++js) {
        qf[64 * js + lane] = make_uint2(hb[js][0], hb[js][1]);
        qf[64 * js + 32 + lane] = make_uint2(lb[js][0], lb[js][1]);
      }
    }
    __syncthreads();
  }
  float qs[NG][2];
  if constexpr (C::KPT) {
#pragma unroll
    for (int gi = 0; gi < NG; ++gi)
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) qs[gi][hh] = qs_s[(2 * c + hh) * NG + gi];
  }
  // scores of quantised caches come out times 2^-24
  const float sig = a.sig_log2 * (C::QUANT ? kCodeScale : 1.f);

  float acc[KS][4];
#pragma unroll
  for (int m = 0; m < KS; ++m) acc[m][0] = acc[m][1] = acc[m][2] = acc[m][3] = 0.f;
  // running maxima start finite, so that 2^(x - m) needs no guard: masked
  // scores are -inf and give 0, and the first live tile replaces the start
  // value (its rescale factor 2^(-1e30 - m) is 0)
  float m_run[2] = {-1e30f, -1e30f}, l_run[2] = {0.f, 0.f};
  float zacc[NG][2];
#pragma unroll
  for (int gi = 0; gi < NG; ++gi) zacc[gi][0] = zacc[gi][1] = 0.f;

  // shared-memory addresses of the fragments (raw records or planes).
  // Symmetric records are rotated as a whole by sym_rot(row); the rows a
  // lane reads for keys are g and g + 8 of a 16-row block, so the rotation
  // is one per lane.
  const int krot = C::SYM ? sym_rot(g, C::NCH) : 0;
  auto k_chunk = [&](const uint8_t *st, int t, int i) -> const uint8_t * {
    if constexpr (C::SYM) return st + t * C::REC + 16 * ((4 * i + c + krot) & (C::NCH - 1));
    else if constexpr (C::TMA) return st + t * C::REC + 16 * (4 * i + c);
    else return st + C::KP_OFF + t * C::KSTR + 16 * kswz(C::KSWZ, t, 4 * i + c);
  };
  auto k_half = [&](const uint8_t *st, int t) -> const uint8_t * {  // 8-byte lane segment
    if constexpr (C::SYM)
      return st + t * C::REC + 16 * (((c >> 1) + krot) & (C::NCH - 1)) + 8 * (c & 1);
    else if constexpr (C::TMA) return st + t * C::REC + 8 * c;
    else return st + C::KP_OFF + t * C::KSTR + 8 * c;
  };
  // symmetric scales of shared-memory row t: (K scale, V scale)
  auto sc_pair = [&](const uint8_t *st, int t) -> float2 {
    const uint32_t w = reinterpret_cast<const uint32_t *>(st + C::SC_OFF_T)[t];
    return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
  };
  auto v_chunk = [&](const uint8_t *st, int t, int k) -> const uint8_t * {
    const int u = g * (C::SV / 16) + k;
    if constexpr (C::TMA) return st + t * C::REC + C::KB + 16 * u;
    else return st + C::VP_OFF + t * C::VSTR + 16 * vswz(C::VSWZ, t, u);
  };
  auto km_row = [&](const uint8_t *st, int t) -> const float2 * {
    if constexpr (C::TMA) return reinterpret_cast<const float2 *>(st + t * C::REC + 2 * C::KB);
    else return reinterpret_cast<const float2 *>(st + C::KM_OFF + t * C::MB);
  };
  auto vm_row = [&](const uint8_t *st, int t) -> const float2 * {
    if constexpr (C::TMA)
      return reinterpret_cast<const float2 *>(st + t * C::REC + 2 * C::KB + (C::KPT ? C::MB : 0));
    else return reinterpret_cast<const float2 *>(st + C::VM_OFF + t * C::MB);
  };
  auto kg_rows = [&](const uint8_t *st) -> const float2 * {
    if constexpr (C::TMA) return reinterpret_cast<const float2 *>(st + C::KG_OFF_T);
    else return reinterpret_cast<const float2 *>(st + C::KG_OFF);
  };

  // ---- per-channel keys: the query folded with the key scales -------------
  // For each group slot of the tile, head n's query times the group's
  // per-channel scales, split hi/lo f16 in the B-fragment order of the score
  // MMA (k-step js, lane), plus each warp's share of sum_ch q[n][ch]
  // zero[ch].  Built once per tile by all threads (every block of a group
  // reads it) instead of by every warp for its own block.  Slots of groups
  // that are not complete hold garbage that no block reads (those rows are
  // scored from the bf16 residual).
  uint4 *fold = reinterpret_cast<uint4 *>(smem + C::FOLD_OFF);
  float *zred = reinterpret_cast<float *>(smem + C::FOLD_OFF + C::FOLD_BYTES);
  auto fold_query = [&](int s) {
    static_assert(!C::KPC || KS % 4 == 0, "k-steps split evenly over the four warps");
    const float2 *kg0 = kg_rows(stages + s * C::STAGE);
    float zp[C::KPC ? C::KG_ROWS : 1];
#pragma unroll
    for (int gs = 0; gs < (C::KPC ? C::KG_ROWS : 1); ++gs) zp[gs] = 0.f;
#pragma unroll
    for (int k = 0; k < C::KG_ROWS * KS / 4; ++k) {
      const int gs = (4 * k) / KS, js = warp + (4 * k) % KS;
      const float *qh = q_s + g * QSTR + 16 * js;
      const float2 *sz = kg0 + gs * D + 16 * js;
      float x[4];
      const int chs[4] = {2 * c, 2 * c + 1, 2 * c + 8, 2 * c + 9};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 m2 = sz[chs[e]];
        zp[gs] += qh[chs[e]] * m2.y;
        x[e] = qh[chs[e]] * m2.x;
        if (BITS == 4 && e >= 2) x[e] *= 0.0625f;
      }
      uint32_t h0, l0, h1, l1;
      split2<false>(x[0], x[1], h0, l0);
      split2<false>(x[2], x[3], h1, l1);
      fold[(gs * KS + js) * 32 + lane] = make_uint4(h0, h1, l0, l1);
    }
#pragma unroll
    for (int gs = 0; gs < (C::KPC ? C::KG_ROWS : 1); ++gs) {
      float z = zp[gs];
      z += __shfl_xor_sync(0xffffffffu, z, 1);
      z += __shfl_xor_sync(0xffffffffu, z, 2);
      if (c == 0 && C::KPC) zred[(warp * C::KG_ROWS + gs) * 8 + g] = z;
    }
  };

  // ---- consumer: one warp's RB blocks of 16 rows of one stage ------------
  constexpr int RB = C::RB;
  auto compute = [&](int t, int s) {
    const int base = i0 + t * C::TILE;
    const int wr0 = 16 * RB * warp;
    if (base + wr0 >= i1) return;  // warp-uniform: no live row
    const uint8_t *st = stages + s * C::STAGE;

    // lane's K words of one row
    auto load_k = [&](int t, uint32_t(&w)[C::NWK]) {
      if constexpr (C::SK >= 16) {
#pragma unroll
        for (int i = 0; i < C::SK / 16; ++i) {
          const uint4 x = *reinterpret_cast<const uint4 *>(k_chunk(st, t, i));
          w[4 * i] = x.x; w[4 * i + 1] = x.y; w[4 * i + 2] = x.z; w[4 * i + 3] = x.w;
        }
      } else {
        const uint2 x = *reinterpret_cast<const uint2 *>(k_half(st, t));
        w[0] = x.x; w[1] = x.y;
      }
    };
    // A fragment registers (a0..a3) of k-step js from the two rows' words
    auto kfrag = [&](const uint32_t(&wa)[C::NWK], const uint32_t(&wb)[C::NWK], int js,
                     uint32_t &a0, uint32_t &a1, uint32_t &a2, uint32_t &a3) {
      if constexpr (BITS == 16) {
        a0 = wa[2 * js]; a2 = wa[2 * js + 1]; a1 = wb[2 * js]; a3 = wb[2 * js + 1];
      } else if constexpr (BITS == 8) {
        a0 = u8pair_f16(wa[js], 0x4140); a2 = u8pair_f16(wa[js], 0x4342);
        a1 = u8pair_f16(wb[js], 0x4140); a3 = u8pair_f16(wb[js], 0x4342);
      } else if constexpr (BITS == 2) {
        // k-step js: byte (js/2) % 2 of each half, fields 2 (js % 2) + {0, 1}
        const int sh = (js & 2) * 4;
        const uint32_t xa = wa[js >> 2] >> sh, xb = wb[js >> 2] >> sh;
        const uint32_t m0 = 0x00030003u << (4 * (js & 1)), m2 = 0x000C000Cu << (4 * (js & 1));
        a0 = xa & m0; a2 = xa & m2;
        a1 = xb & m0; a3 = xb & m2;
      } else {
        const int sh = (js & 1) * 8;
        const uint32_t xa = wa[js >> 1] >> sh, xb = wb[js >> 1] >> sh;
        a0 = nib_f16(xa, 0x000F000Fu); a2 = nib_f16(xa, 0x00F000F0u);
        a1 = nib_f16(xb, 0x000F000Fu); a3 = nib_f16(xb, 0x00F000F0u);
      }
    };

    // ---- scores of each 16-row block (raw dot products, fp32) --------------
    float s4[RB][4];
    bool vA[RB], vB[RB];
#pragma unroll
    for (int rb = 0; rb < RB; ++rb) {
      const int r0 = wr0 + 16 * rb;
      const int tA = r0 + g, tB = tA + 8;
      vA[rb] = base + tA < i1;
      vB[rb] = base + tB < i1;
      if constexpr (C::TMA) {
        if (gather) {
          constexpr int RPW = C::TILE / 4;
          vA[rb] = (gmask[s * 4 + tA / RPW] >> (tA % RPW)) & 1u;
          vB[rb] = (gmask[s * 4 + tB / RPW] >> (tB % RPW)) & 1u;
        }
      } else if (gather) {
        if (vA[rb]) { const int p = kept[base + tA]; vA[rb] = p >= 0 && p < len; }
        if (vB[rb]) { const int p = kept[base + tB]; vB[rb] = p >= 0 && p < len; }
      }
      s4[rb][0] = s4[rb][1] = s4[rb][2] = s4[rb][3] = 0.f;
      if (base + r0 >= i1) continue;
      if (C::KPC && base + r0 >= Tq) {
        // open per-channel key group (at most group-1 positions): bf16 rows
        // of the residual plane, stored in the bf16 K fragment order, read
        // from global memory straight into A fragments; the query enters as
        // bf16 hi + lo fragments, fp32 accumulation.
        const uint8_t *res = v.resid + slab * (size_t)GS * D * 2;
        const uint8_t *rowA = res + (size_t)((base + tA) % GS) * D * 2;
        const uint8_t *rowB = res + (size_t)((base + tB) % GS) * D * 2;
        float d[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int i = 0; i < D / 32; ++i) {
          const uint4 z = make_uint4(0, 0, 0, 0);
          const uint4 xa = vA[rb] ? *reinterpret_cast<const uint4 *>(rowA + 16 * (4 * i + c)) : z;
          const uint4 xb = vB[rb] ? *reinterpret_cast<const uint4 *>(rowB + 16 * (4 * i + c)) : z;
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const float *qh = q_s + g * QSTR + 16 * (2 * i + h);
            uint32_t b0, b0l, b1, b1l;
            split2<true>(qh[2 * c], qh[2 * c + 1], b0, b0l);
            split2<true>(qh[2 * c + 8], qh[2 * c + 9], b1, b1l);
            const uint32_t a0 = h ? xa.z : xa.x, a2 = h ? xa.w : xa.y;
            const uint32_t a1 = h ? xb.z : xb.x, a3 = h ? xb.w : xb.y;
            mma_bf16(d, a0, a1, a2, a3, b0, b1);
            mma_bf16(d, a0, a1, a2, a3, b0l, b1l);
          }
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) s4[rb][k] = d[k] * kCodeUnit;  // scores carry 2^-24
      } else if constexpr (C::KPC) {
        // the query folded with this group's per-channel scales (built for
        // the tile by fold_query), the zero points entering as one per-head
        // constant in the 2^-24 units of the MMA
        const int gs = r0 / GS;
        const uint4 *fg = fold + gs * KS * 32 + lane;
        float2 z2 = make_float2(0.f, 0.f);
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const float2 zw = *reinterpret_cast<const float2 *>(zred + (w * C::KG_ROWS + gs) * 8 + 2 * c);
          z2.x += zw.x;
          z2.y += zw.y;
        }
        const float corr0 = z2.x * kCodeUnit, corr1 = z2.y * kCodeUnit;
        uint32_t wa[C::NWK], wb[C::NWK];
        load_k(tA, wa);
        load_k(tB, wb);
        // hi and lo products in two accumulator chains
        float d[4] = {corr0, corr1, corr0, corr1}, dl[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int js = 0; js < KS; ++js) {
          uint32_t a0, a1, a2, a3;
          kfrag(wa, wb, js, a0, a1, a2, a3);
          const uint4 f = fg[js * 32];
          mma_f16(d, a0, a1, a2, a3, f.x, f.y);
          mma_f16(dl, a0, a1, a2, a3, f.z, f.w);
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) s4[rb][k] = d[k] + dl[k];
      } else {
        uint32_t wa[C::NWK], wb[C::NWK];
        load_k(tA, wa);
        load_k(tB, wb);
        if constexpr (BF) {
          float d[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int js = 0; js < KS; ++js) {
            uint32_t a0, a1, a2, a3;
            kfrag(wa, wb, js, a0, a1, a2, a3);
            const uint2 qh = qf[64 * js + lane];
            mma_bf16(d, a0, a1, a2, a3, qh.x, qh.y);
            if (use_lo) {
              const uint2 ql = qf[64 * js + 32 + lane];
              mma_bf16(d, a0, a1, a2, a3, ql.x, ql.y);
            }
          }
#pragma unroll
          for (int k = 0; k < 4; ++k) s4[rb][k] = d[k];
        } else {
          const float2 *kmA = km_row(st, tA);
          const float2 *kmB = km_row(st, tB);
          constexpr int JPG = GS / 16;  // k-steps per group
          float4 qA, qB;  // (scale, zero) of groups 2j and 2j + 1: one 16-byte load
          if constexpr (C::SYM) {  // one group: scale s, zero -q s
            const float kA = sc_pair(st, tA).x, kB = sc_pair(st, tB).x;
            qA = make_float4(kA, -C::QL * kA, 0.f, 0.f);
            qB = make_float4(kB, -C::QL * kB, 0.f, 0.f);
          }
#pragma unroll
          for (int gi = 0; gi < NG; ++gi) {
            if (!C::SYM && (gi & 1) == 0) {
              qA = reinterpret_cast<const float4 *>(kmA)[gi >> 1];
              qB = reinterpret_cast<const float4 *>(kmB)[gi >> 1];
            }
            // long groups accumulate alternate k-steps in two chains
            constexpr int NCHAIN = JPG >= 4 ? 2 : 1;
            float dd[NCHAIN][4];
#pragma unroll
            for (int h = 0; h < NCHAIN; ++h) dd[h][0] = dd[h][1] = dd[h][2] = dd[h][3] = 0.f;
#pragma unroll
            for (int jj = 0; jj < JPG; ++jj) {
              const int js = gi * JPG + jj;
              uint32_t a0, a1, a2, a3;
              kfrag(wa, wb, js, a0, a1, a2, a3);
              const uint2 qh = qf[64 * js + lane];
              mma_f16(dd[jj % NCHAIN], a0, a1, a2, a3, qh.x, qh.y);
              if (use_lo) {
                const uint2 ql = qf[64 * js + 32 + lane];
                mma_f16(dd[jj % NCHAIN], a0, a1, a2, a3, ql.x, ql.y);
              }
            }
            float d[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) d[k] = NCHAIN == 2 ? dd[0][k] + dd[NCHAIN - 1][k] : dd[0][k];
            const float2 mA = (gi & 1) ? make_float2(qA.z, qA.w) : make_float2(qA.x, qA.y);
            const float2 mB = (gi & 1) ? make_float2(qB.z, qB.w) : make_float2(qB.x, qB.y);
            s4[rb][0] = fmaf(mA.x, d[0], fmaf(mA.y, qs[gi][0], s4[rb][0]));
            s4[rb][1] = fmaf(mA.x, d[1], fmaf(mA.y, qs[gi][1], s4[rb][1]));
            s4[rb][2] = fmaf(mB.x, d[2], fmaf(mB.y, qs[gi][0], s4[rb][2]));
            s4[rb][3] = fmaf(mB.x, d[3], fmaf(mB.y, qs[gi][1], s4[rb][3]));
          }
        }
      }
    }

    // ---- online softmax over the warp's rows (base 2, lazy rescaling) ------
    float p[RB][4];
    float mt0 = -INFINITY, mt1 = -INFINITY;
#pragma unroll
    for (int rb = 0; rb < RB; ++rb) {
      // raw scores here; the scale (> 0, checked by the host) enters the
      // maxima once and the exponent through one FMA
      p[rb][0] = vA[rb] ? s4[rb][0] : -INFINITY;
      p[rb][1] = vA[rb] ? s4[rb][1] : -INFINITY;
      p[rb][2] = vB[rb] ? s4[rb][2] : -INFINITY;
      p[rb][3] = vB[rb] ? s4[rb][3] : -INFINITY;
      mt0 = fmaxf(mt0, fmaxf(p[rb][0], p[rb][2]));
      mt1 = fmaxf(mt1, fmaxf(p[rb][1], p[rb][3]));
    }
    // Keep a stale maximum while every score of the tile stays within 2^8
    // of it: the result is exact either way.  One vote decides; only tiles
    // that raise some lane's maximum reduce it over the row lanes and
    // rescale.
    mt0 *= sig;
    mt1 *= sig;
    const bool need = (mt0 > m_run[0] + 8.f) || (mt1 > m_run[1] + 8.f);
    if (__any_sync(0xffffffffu, need)) {
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
        mt0 = fmaxf(mt0, __shfl_xor_sync(0xffffffffu, mt0, off));
        mt1 = fmaxf(mt1, __shfl_xor_sync(0xffffffffu, mt1, off));
      }
      const float n0 = fmaxf(m_run[0], mt0), n1 = fmaxf(m_run[1], mt1);
      const float al0 = fast_exp2(m_run[0] - n0);
      const float al1 = fast_exp2(m_run[1] - n1);
#pragma unroll
      for (int m = 0; m < KS; ++m) {
        acc[m][0] *= al0; acc[m][2] *= al0;
        acc[m][1] *= al1; acc[m][3] *= al1;
      }
      l_run[0] *= al0; l_run[1] *= al1;
#pragma unroll
      for (int gi = 0; gi < NG; ++gi) { zacc[gi][0] *= al0; zacc[gi][1] *= al1; }
      m_run[0] = n0; m_run[1] = n1;
    }
    {
#pragma unroll
      for (int rb = 0; rb < RB; ++rb) {
        p[rb][0] = fast_exp2(fmaf(p[rb][0], sig, -m_run[0]));
        p[rb][1] = fast_exp2(fmaf(p[rb][1], sig, -m_run[1]));
        p[rb][2] = fast_exp2(fmaf(p[rb][2], sig, -m_run[0]));
        p[rb][3] = fast_exp2(fmaf(p[rb][3], sig, -m_run[1]));
        l_run[0] += p[rb][0] + p[rb][2];
        l_run[1] += p[rb][1] + p[rb][3];
      }
    }

    // ---- value product: A = V^T from the lanes' segments of 4 positions ----
    if constexpr (BITS == 16) {
#pragma unroll
      for (int rb = 0; rb < RB; ++rb) {
        const int r0 = wr0 + 16 * rb;
        if (base + r0 >= i1) continue;
        // P^T fragments: P split hi/lo, transposed from the score layout
        uint32_t pf[4];
        {
          uint32_t ht, lt, hb, lb;
          split2<true>(p[rb][0], p[rb][1], ht, lt);
          split2<true>(p[rb][2], p[rb][3], hb, lb);
          pf[0] = movmatrix_t(ht); pf[1] = movmatrix_t(hb);
          pf[2] = movmatrix_t(lt); pf[3] = movmatrix_t(lb);
        }
        const int T0 = r0 + 2 * c, T1 = T0 + 1, T2 = T0 + 8, T3 = T0 + 9;
        // one word per M-block: (row g, row g+8) of one position
#pragma unroll
        for (int k = 0; k < C::SV / 16; ++k) {
          const uint4 w0 = *reinterpret_cast<const uint4 *>(v_chunk(st, T0, k));
          const uint4 w1 = *reinterpret_cast<const uint4 *>(v_chunk(st, T1, k));
          const uint4 w2 = *reinterpret_cast<const uint4 *>(v_chunk(st, T2, k));
          const uint4 w3 = *reinterpret_cast<const uint4 *>(v_chunk(st, T3, k));
          const uint32_t x0[4] = {w0.x, w0.y, w0.z, w0.w}, x1[4] = {w1.x, w1.y, w1.z, w1.w};
          const uint32_t x2[4] = {w2.x, w2.y, w2.z, w2.w}, x3[4] = {w3.x, w3.y, w3.z, w3.w};
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const int m = 4 * k + q;
            const uint32_t a0 = __byte_perm(x0[q], x1[q], 0x5410);
            const uint32_t a1 = __byte_perm(x0[q], x1[q], 0x7632);
            const uint32_t a2 = __byte_perm(x2[q], x3[q], 0x5410);
            const uint32_t a3 = __byte_perm(x2[q], x3[q], 0x7632);
            mma_bf16(acc[m], a0, a1, a2, a3, pf[0], pf[1]);
            mma_bf16(acc[m], a0, a1, a2, a3, pf[2], pf[3]);
          }
        }
      }
    } else {
      // Value codes by ldmatrix.trans: matrix (j, k) is chunk k of the 8
      // positions 16 rb + 8 j + i of the row block; lane (g, c) receives
      // element g of positions 2c and 2c+1, i.e. its bytes of M-blocks
      // (2k, 2k+1) (4-bit) or of M-block k (8-bit) for both positions.
      // Chunks are stored rotated by v_rot(position) (conflict-free rows).
      constexpr int NC = C::KB / 16;  // value chunks per record
      uint32_t vw[RB][2 * NC];        // [rb][NC j + k]
#pragma unroll
      for (int rb = 0; rb < RB; ++rb) {
#pragma unroll
        for (int q = 0; q < NC / 2; ++q) {
          const int mi = 4 * q + (lane >> 3);  // this lane addresses matrix mi
          const int j = mi / NC, k = mi % NC;
          const int t = wr0 + 16 * rb + 8 * j + (lane & 7);
          // rotation of the row's record: by its shared-memory row, or (row
          // gather) by its position, read from the stage's rotation bytes
          const int vr = (C::GTMA && gather) ? rotb[s * C::TILE + t] : v_rot(t, C::REC, NC);
          const uint8_t *src =
              C::SYM ? st + t * C::REC + 16 * ((NC + k + sym_rot(t, C::NCH)) & (C::NCH - 1))
                     : st + t * C::REC + C::KB + 16 * ((k + vr) & (NC - 1));
          ldmatrix_x4_t(vw[rb][4 * q], vw[rb][4 * q + 1], vw[rb][4 * q + 2], vw[rb][4 * q + 3],
                        src);
        }
      }
      uint32_t pf[RB][4];
      float4 vA4[RB], vB4[RB];  // (scale, zero) of groups 2j, 2j + 1 of rows g, g + 8
      // M-blocks in pairs (groups span whole pairs): the four MMAs of a
      // pair and row block alternate between the two accumulators
      static_assert(GS % 32 == 0, "value groups cover whole M-block pairs");
#pragma unroll
      for (int m0 = 0; m0 < KS; m0 += 2) {
        const int gi = (16 * m0) / GS;
        if ((16 * m0) % GS == 0) {
          // P' = p * value scale of this channel group, split hi/lo and
          // transposed; the zero points accumulate separately.
#pragma unroll
          for (int rb = 0; rb < RB; ++rb) {
            const int tA = wr0 + 16 * rb + g;
            if constexpr (C::SYM) {
              // rows without a position have p = 0 but possibly a stale
              // scale word: their scale becomes 0 (0 * NaN would poison)
              const float sA = vA[rb] ? sc_pair(st, tA).y : 0.f;
              const float sB = vB[rb] ? sc_pair(st, tA + 8).y : 0.f;
              vA4[rb] = make_float4(sA, -C::QL * sA, 0.f, 0.f);
              vB4[rb] = make_float4(sB, -C::QL * sB, 0.f, 0.f);
            } else if ((gi & 1) == 0) {
              vA4[rb] = reinterpret_cast<const float4 *>(vm_row(st, tA))[gi >> 1];
              vB4[rb] = reinterpret_cast<const float4 *>(vm_row(st, tA + 8))[gi >> 1];
              if constexpr (C::GTMA && gather) {
                // rows without a position hold another record's bytes
                // (p = 0 there, but 0 * a non-finite scale would poison)
                if (!vA[rb]) vA4[rb] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (!vB[rb]) vB4[rb] = make_float4(0.f, 0.f, 0.f, 0.f);
              }
            }
            const float2 mA = (gi & 1) ? make_float2(vA4[rb].z, vA4[rb].w)
                                       : make_float2(vA4[rb].x, vA4[rb].y);
            const float2 mB = (gi & 1) ? make_float2(vB4[rb].z, vB4[rb].w)
                                       : make_float2(vB4[rb].x, vB4[rb].y);
            uint32_t ht, lt, hb, lb;
            split2<false>(p[rb][0] * mA.x, p[rb][1] * mA.x, ht, lt);
            split2<false>(p[rb][2] * mB.x, p[rb][3] * mB.x, hb, lb);
            pf[rb][0] = movmatrix_t(ht); pf[rb][1] = movmatrix_t(hb);
            pf[rb][2] = movmatrix_t(lt); pf[rb][3] = movmatrix_t(lb);
            zacc[gi][0] = fmaf(p[rb][0], mA.y, fmaf(p[rb][2], mB.y, zacc[gi][0]));
            zacc[gi][1] = fmaf(p[rb][1], mA.y, fmaf(p[rb][3], mB.y, zacc[gi][1]));
          }
        }
#pragma unroll
        for (int rb = 0; rb < RB; ++rb) {
          uint32_t af[2][4];
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const int m = m0 + u;
            uint32_t &a0 = af[u][0], &a1 = af[u][1], &a2 = af[u][2], &a3 = af[u][3];
            if constexpr (BITS == 8) {
              // bytes (row g, row g+8) of the two positions: (0, 2) and (1, 3)
              const uint32_t X0 = vw[rb][m], X2 = vw[rb][NC + m];
              a0 = u8pair_f16(X0, 0x4240); a1 = u8pair_f16(X0, 0x4341);
              a2 = u8pair_f16(X2, 0x4240); a3 = u8pair_f16(X2, 0x4341);
            } else if constexpr (BITS == 2) {
              // byte (m/2) % 2 of each half, field 2 (m % 2) (row g) and
              // 2 (m % 2) + 1 (row g+8): weights 4^(2 (m%2)) and 4^(2 (m%2) + 1)
              const int sh = (m & 2) * 4;
              const uint32_t X0 = vw[rb][m >> 2] >> sh, X2 = vw[rb][NC + (m >> 2)] >> sh;
              const uint32_t mg = 0x00030003u << (4 * (m & 1)), mh = 0x000C000Cu << (4 * (m & 1));
              a0 = X0 & mg; a1 = X0 & mh;
              a2 = X2 & mg; a3 = X2 & mh;
            } else {
              // bytes 0 and 2 (even m) or 1 and 3 (odd m): row g in the low
              // nibble, row g+8 in the high nibble (16x, undone at the end)
              const int sh = 8 * (m & 1);
              const uint32_t X0 = vw[rb][m >> 1] >> sh, X2 = vw[rb][NC + (m >> 1)] >> sh;
              a0 = nib_f16(X0, 0x000F000Fu); a1 = nib_f16(X0, 0x00F000F0u);
              a2 = nib_f16(X2, 0x000F000Fu); a3 = nib_f16(X2, 0x00F000F0u);
            }
          }
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int u = 0; u < 2; ++u)
              mma_f16(acc[m0 + u], af[u][0], af[u][1], af[u][2], af[u][3], pf[rb][2 * h],
                      pf[rb][2 * h + 1]);
        }
      }
    }
  };

  // ---- copy ring over the split's tiles -----------------------------------
  bool timed_out = false;
  int t_stop = n_tiles;  // first tile not consumed
  // Bulk-copy ring (quantised per-token keys, contiguous or gathered by row
  // copies): the stage that
  // tile t - 1 used is refilled as soon as every warp has finished it,
  // before tile t is awaited, so NST copies are in flight during each wait.
  // The barrier at the top of an iteration both frees that stage and lets
  // all threads agree whether a wait of the previous iteration gave up
  // (a warp whose wait gave up skips that tile's arithmetic).
  constexpr bool kEarly = C::TMA && !C::KPC && (!gather || C::GTMA);
  if constexpr (kEarly) {
    bool ok = true;
    int t_fail = -1;
    for (int t = 0; t < n_tiles; ++t) {
      if (__syncthreads_or(!ok)) {
        t_fail = t - 1;
        break;
      }
      const int nt = t + C::NST - 1;
      if (nt < n_tiles) issue(nt, nt % C::NST);
      ok = __all_sync(0xffffffffu, mbar_wait(&bars[t % C::NST], (t / C::NST) & 1, a.wait_limit));
      if (ok) compute(t, t % C::NST);
    }
    if (t_fail < 0 && __syncthreads_or(!ok)) t_fail = n_tiles - 1;
    if (t_fail >= 0) {
      timed_out = true;
      if (tid == 0) set_err(a.err, 8);
      // tiles t_fail .. t_fail + NST - 1 were issued: let them land (bounded)
      const int t_end = min(n_tiles, t_fail + C::NST);
      for (int u = t_fail; u < t_end; ++u) mbar_wait(&bars[u % C::NST], (u / C::NST) & 1, 1u << 20);
    }
  } else {
    for (int t = 0; t < n_tiles; ++t) {
      bool ok = true;
      if (use_cp)
        cp_async_wait<C::NST - 2>();
      else
        ok = mbar_wait(&bars[t % C::NST], (t / C::NST) & 1, a.wait_limit);
      // every thread has finished tile t-1, and all agree whether a wait gave up
      if (__syncthreads_or(!ok)) {
        timed_out = true;
        t_stop = t;
        if (tid == 0) set_err(a.err, 8);
        break;
      }
      const int nt = t + C::NST - 1;
      if (nt < n_tiles) issue(nt, nt % C::NST);
      if (use_cp) cp_async_commit();
      if constexpr (C::KPC) {
        fold_query(t % C::NST);
        __syncthreads();
      }
      compute(t, t % C::NST);
    }
    if (!use_cp) {
      if (timed_out) {
        // let copies still in flight land (bounded) before the CTA leaves:
        // tiles t_stop .. t_stop + NST - 2 were issued and not consumed
        const int t_end = min(n_tiles, t_stop + C::NST - 1);
        for (int u = t_stop; u < t_end; ++u) mbar_wait(&bars[u % C::NST], (u / C::NST) & 1, 1u << 20);
      }
    } else {
      cp_async_wait<0>();
    }
  }
  __syncthreads();

  pdl_trigger();  // the next kernel may be scheduled as this grid retires

  // ---- finish this warp's state ------------------------------------------
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
    l_run[0] += __shfl_xor_sync(0xffffffffu, l_run[0], off);
    l_run[1] += __shfl_xor_sync(0xffffffffu, l_run[1], off);
#pragma unroll
    for (int gi = 0; gi < NG; ++gi) {
      zacc[gi][0] += __shfl_xor_sync(0xffffffffu, zacc[gi][0], off);
      zacc[gi][1] += __shfl_xor_sync(0xffffffffu, zacc[gi][1], off);
    }
  }
  float *red = reinterpret_cast<float *>(stages);  // [4 warps][8 heads][D + 2]
  constexpr int RS = D + 2;
#pragma unroll
  for (int m = 0; m < KS; ++m) {
    const int ch0 = 16 * m + g, ch1 = ch0 + 8;
    const int gi = C::QUANT ? (16 * m) / GS : 0;
    constexpr float vsc = C::QUANT ? kCodeScale : 1.f;  // value codes carry 2^-24
    // code weights of rows g and g+8 of M-block m, undone here
    const float ls = (BITS == 2 && (m & 1)) ? 0.0625f * vsc : vsc;
    const float hs = (BITS == 4) ? 0.0625f * vsc
                   : (BITS == 2) ? ((m & 1) ? 0.015625f * vsc : 0.25f * vsc) : vsc;
    const float z0 = C::QUANT ? zacc[gi][0] : 0.f, z1 = C::QUANT ? zacc[gi][1] : 0.f;
    red[(warp * 8 + 2 * c) * RS + ch0] = acc[m][0] * ls + z0;
    red[(warp * 8 + 2 * c + 1) * RS + ch0] = acc[m][1] * ls + z1;
    red[(warp * 8 + 2 * c) * RS + ch1] = acc[m][2] * hs + z0;
    red[(warp * 8 + 2 * c + 1) * RS + ch1] = acc[m][3] * hs + z1;
  }
  if (g == 0) {
    red[(warp * 8 + 2 * c) * RS + D] = m_run[0];
    red[(warp * 8 + 2 * c) * RS + D + 1] = l_run[0];
    red[(warp * 8 + 2 * c + 1) * RS + D] = m_run[1];
    red[(warp * 8 + 2 * c + 1) * RS + D + 1] = l_run[1];
  }
  __syncthreads();

  // ---- merge the four warps; write output or split partial ---------------
  const size_t row0 = (size_t)b * a.Hq + (size_t)kvh * a.G;
  for (int h = 0; h < a.G; ++h) {
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) M = fmaxf(M, red[(w * 8 + h) * RS + D]);
    float wt[4], L = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float mw = red[(w * 8 + h) * RS + D];
      wt[w] = (mw == -INFINITY || M == -INFINITY) ? 0.f : exp2f(mw - M);
      L += wt[w] * red[(w * 8 + h) * RS + D + 1];
    }
    for (int ch = tid; ch < D; ch += 128) {
      float A = 0.f;
#pragma unroll
      for (int w = 0; w < 4; ++w) A += wt[w] * red[(w * 8 + h) * RS + ch];
      if (a.out) {
        a.out[(row0 + h) * D + ch] = (L > 0.f) ? A / L : 0.f;
      } else {
        float *pr = a.partial + ((size_t)slot * v.B * a.Hq + row0 + h) * RS;
        pr[ch] = A;
        if (ch == 0) { pr[D] = (L > 0.f) ? M : -INFINITY; pr[D + 1] = L; }
      }
    }
  }
  return !timed_out;
}

// Formats with a run-schedule kernel: the contiguous bulk-copy formats
// (quantised, per-token keys or the symmetric scheme).
template <int BITS, int D, int KAX, int GS>
__host__ __device__ constexpr bool gqa_has_run() {
  using C = GqaCfg<BITS, D, KAX, GS>;
  return C::TMA && !C::KPC;
}

// Segment k (0 or 1) of run-schedule CTA blockIdx.x (see gqa_decode_kernel):
// unit (b, kvh), items [i0, i1) (i1 = -1: to the sequence's end), partial
// slot, and the number of slots the unit's pieces fill when this CTA holds
// its last planned tile (else 0).  False when the run has no segment k.
// Each unit spans a.run_tpu planned tiles of the run grid: a.run_setup
// tiles standing for the cost of starting a unit (query set-up, the first
// copies, the epilogue), then its data tiles, so that a run that starts a
// second unit carries fewer data tiles.  32-bit arithmetic only (the host
// keeps W < 2^31 and n < 2^16): with W = q n + r, run c starts at planned
// tile floor(c W / n) = c q + floor(c r / n).
struct GqaRunSeg {
  int b, kvh, i0, i1, slot, n_used;
};
__device__ __forceinline__ int gqa_run_start(const GqaDecodeArgs &a, int c) {
  return c * a.run_q + (int)(((uint32_t)c * (uint32_t)a.run_r) / (uint32_t)a.run_ctas);
}
template <int TILE>
__device__ __forceinline__ bool gqa_run_segment(const GqaDecodeArgs &a, int k, GqaRunSeg &sg) {
  const int x = blockIdx.x, tpu = a.run_tpu, su = a.run_setup;
  const int w1 = gqa_run_start(a, x + 1);
  int w = gqa_run_start(a, x);
  if (k == 1) w = (w / tpu + 1) * tpu;  // the next unit's first planned tile
  if (w >= w1) return false;
  const int u = w / tpu;
  const int ub = u * tpu, we = min(w1, ub + tpu);
  const bool owns_end = we == ub + tpu;
  // the first CTA whose run meets unit u: this one, or an earlier one whose
  // run holds planned tile ub (runs are at least q >= 1 tiles, so at most a
  // unit's worth of steps back)
  int c0 = x;
  while (gqa_run_start(a, c0) > ub) --c0;
  sg.b = u / a.v.Hkv;
  sg.kvh = u - sg.b * a.v.Hkv;
  sg.i0 = max(0, w - ub - su) * TILE;
  sg.i1 = owns_end ? -1 : max(0, we - ub - su) * TILE;
  sg.slot = x - c0;
  sg.n_used = owns_end ? sg.slot + 1 : 0;
  return true;
}

// RUN = false: grid (split, kv head, sequence); CTA (x, y, z) decodes items
// [x ips, (x + 1) ips) of unit (z, y) into partial slot x (ips =
// a.items_per_split; the last split runs to the end, so a launch recorded
// for shorter sequences, as in a replayed graph, still covers every
// position).
// RUN = true: a one-dimensional grid of equal runs.  The (unit, tile) grid,
// u = b Hkv + kvh with a.run_tpu planned tiles each (set-up tiles, then
// data tiles), is flattened and CTA x takes planned tiles [w0, w1), w0 =
// floor(x W / n) (W tiles, n CTAs).  The host
// keeps runs no longer than a unit, so a run meets at most two units; each
// is one segment, decoded into partial slot x - (the first CTA meeting the
// unit), each on its own set of mbarriers.  The CTA that holds a unit's
// last planned tile runs to the sequence's end and marks the unit's unused
// slots (up to a.run_slots) empty.  Every CTA does
// W / n tiles of work, so one wave of resident CTAs ends together instead
// of a second, partial wave of splits.
template <int BITS, int D, int KAX, int GS, bool GATHER, bool RUN>
__global__ void __launch_bounds__(128, GqaCfg<BITS, D, KAX, GS>::MIN_CTAS)
    gqa_decode_kernel(const __grid_constant__ CUtensorMap rows, const GqaDecodeArgs a) {
  pdl_wait();
  using C = GqaCfg<BITS, D, KAX, GS>;
  extern __shared__ __align__(128) uint8_t smem[];
  if constexpr (GATHER && C::GTMA) {
    // row-copy destinations are 128-byte aligned relative to the base
    if (smem_u32(smem) & 127u) {
      if (threadIdx.x == 0) set_err(a.err, 16);  // KVK_DEVERR_ALIGN
      return;
    }
  }
  if constexpr (C::TMA) {
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + C::BAR_OFF);
    if (threadIdx.x == 0) {
#pragma unroll
      for (int s = 0; s < (RUN ? 2 : 1) * C::NST; ++s) mbar_init(&bars[s], 1);
      fence_mbar_init();
    }
    __syncthreads();
  }
  if constexpr (!RUN) {
    const int split = blockIdx.x;
    const int i0 = split * a.items_per_split;
    const int i1 = split == a.n_splits - 1 ? -1 : i0 + a.items_per_split;
    gqa_decode_unit<BITS, D, KAX, GS, GATHER>(a, &rows, blockIdx.z, blockIdx.y, i0, i1, split, 0);
  } else {
    static_assert(gqa_has_run<BITS, D, KAX, GS>() && !GATHER, "runs cover the contiguous bulk-copy formats");
    // Every thread derives the segments from blockIdx.x and the arguments
    // alone (warp-uniform values, as the split grid's are), the second one
    // after the first segment.  The two segments are two call sites, not a
    // loop: inside a loop the decode body compiles to slower code.
    auto mark_unused = [&](const GqaRunSeg &sg) {
      if (sg.n_used == 0) return;
      // slots past the unit's last CTA, for its G heads: whole empty rows
      // (accumulator 0, m = -inf, l = 0), like a split that reads nothing
      const size_t row0 = (size_t)sg.b * a.Hq + (size_t)sg.kvh * a.G;
      constexpr int RS = D + 2;
      for (int i = threadIdx.x; i < (a.run_slots - sg.n_used) * a.G * RS; i += blockDim.x) {
        const int r = i / RS, col = i - r * RS;
        float *pr = a.partial + ((size_t)(sg.n_used + r / a.G) * a.v.B * a.Hq + row0 + r % a.G) * RS;
        pr[col] = col == D ? -INFINITY : 0.f;
      }
    };
    GqaRunSeg sg;
    if (!gqa_run_segment<C::TILE>(a, 0, sg)) return;
    // false: a wait gave up (the error word is set)
    if (!gqa_decode_unit<BITS, D, KAX, GS, false>(a, &rows, sg.b, sg.kvh, sg.i0, sg.i1, sg.slot, 0))
      return;
    mark_unused(sg);
    if (!gqa_run_segment<C::TILE>(a, 1, sg)) return;
    __syncthreads();  // the next unit's query and copies reuse shared memory
    if (!gqa_decode_unit<BITS, D, KAX, GS, false>(a, &rows, sg.b, sg.kvh, sg.i0, sg.i1, sg.slot, 1))
      return;
    mark_unused(sg);
  }
}

template <int BITS, int D, int KAX, int GS, bool GATHER, bool RUN>
cudaError_t launch_gqa_decode_g(const GqaDecodeArgs &a, cudaStream_t st) {
  using C = GqaCfg<BITS, D, KAX, GS>;
  auto k = gqa_decode_kernel<BITS, D, KAX, GS, GATHER, RUN>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  // the record table's tensor map (row gather), else an unused zero map
  CUtensorMap rows;
  memset(&rows, 0, sizeof rows);
  if (GATHER && C::GTMA) {
    if (!a.rows) return cudaErrorInvalidValue;
    memcpy(&rows, a.rows, sizeof rows);
  }
  if constexpr (RUN) return launch_pdl(k, dim3(a.run_ctas), dim3(128), C::SMEM, st, rows, a);
  dim3 grid(a.n_splits, a.v.Hkv, a.v.B);
  return launch_pdl(k, grid, dim3(128), C::SMEM, st, rows, a);
}

template <int BITS, int D, int KAX, int GS>
cudaError_t launch_gqa_decode_t(const GqaDecodeArgs &a, cudaStream_t st) {
  if (a.run_ctas > 0) {
    // run schedule: contiguous bulk-copy formats, partials only
    if constexpr (gqa_has_run<BITS, D, KAX, GS>()) {
      if (a.gather || a.out || a.run_tpu < 1 || a.run_slots < 1) return cudaErrorInvalidValue;
      return launch_gqa_decode_g<BITS, D, KAX, GS, false, true>(a, st);
    } else {
      return cudaErrorInvalidValue;
    }
  }
  if constexpr (GqaCfg<BITS, D, KAX, GS>::KPC) {
    if (a.gather) return cudaErrorInvalidValue;  // no kept lists with per-channel keys
    return launch_gqa_decode_g<BITS, D, KAX, GS, false, false>(a, st);
  } else {
    return a.gather ? launch_gqa_decode_g<BITS, D, KAX, GS, true, false>(a, st)
                    : launch_gqa_decode_g<BITS, D, KAX, GS, false, false>(a, st);
  }
}


template <int BITS, int D, int KAX, int GS>
int gqa_tile_t() {
  return GqaCfg<BITS, D, KAX, GS>::TILE;
}

template <int BITS, int D, int KAX, int GS>
int gqa_ctas_per_sm_t() {
  using C = GqaCfg<BITS, D, KAX, GS>;
  auto k = gqa_decode_kernel<BITS, D, KAX, GS, false, false>;
  cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k, 128, C::SMEM) != cudaSuccess) n = 1;
  return n > 0 ? n : 1;
}

}  // namespace kvk
