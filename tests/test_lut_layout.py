"""Layout rules of the rotated-table kernel (App. A.1 table order; aq_lut.cu), checked on the
CPU: conflict-free shared-memory banks for every code pattern, the byte-permute address
assembly, and the code-byte rotation (whole 8-byte steps by the order of the ring's slot
reads, then one word select and a funnel shift).  Pure integer arithmetic; no device."""

import pytest

TABLE_ADDR = 0x20000          # shared-window address of the tables (a multiple of 64 KB)
BANKS = 32


def prmt(a, b, sel):
    """PTX prmt.b32 default mode: result byte i = byte (nibble i of sel) & 7 of {a, b}."""
    src = a | (b << 32)
    out = 0
    for i in range(4):
        k = (sel >> (4 * i)) & 7
        out |= ((src >> (8 * k)) & 0xFF) << (8 * i)
    return out


@pytest.mark.parametrize("TP", [1, 2, 4])
def test_phase_lanes_hit_distinct_banks_for_any_codes(TP):
    """Entry e of table t is at word e*64 + t*TP (and its copy at e*64 + (t + NT)*TP).  The
    32/TP lanes of one shared-memory phase (distinct l') read slot l' + s at step s: their
    TP-word entries cover distinct banks whatever the codes e, since e*64 = 0 mod 32."""
    NT = 32 // TP
    for s in range(NT):
        for codes in ([0] * NT, list(range(NT)), [255 - 7 * i for i in range(NT)]):
            banks = []
            for lp in range(NT):
                word = codes[lp] * 64 + (lp + s) * TP
                banks += [(word + w) % BANKS for w in range(TP)]
            assert sorted(banks) == list(range(BANKS))
            assert all(lp + s < 2 * NT for lp in range(NT))     # inside the duplicated slots


@pytest.mark.parametrize("TP", [1, 2, 4])
def test_byte_permute_assembles_the_entry_address(TP):
    """One prmt per lookup: code -> byte 1, the lane's slot offset (byte 0) and the table base
    (byte 2) from lane_reg; the step's offset s*TP*4 is added as an immediate without carrying
    into the code byte."""
    NT = 32 // TP
    for lp in range(NT):
        lane_reg = TABLE_ADDR | (lp * TP * 4)
        assert (lane_reg >> 8) & 0xFF == 0
        for s in range(NT):
            for c in range(4):
                for code in (0, 1, 127, 255):
                    word = code << (8 * c) | (0xA5 << (8 * ((c + 1) % 4)))
                    addr = prmt(word, lane_reg, 0x7604 | (c << 4)) + s * TP * 4
                    assert addr == TABLE_ADDR + code * 256 + (lp + s) * TP * 4
                    assert lp * TP * 4 + s * TP * 4 < 256


def _kernel_rotation(stream_bytes, li, NT, P):
    """The kernel's rotation of a row's NT code bytes by li: the ring holds the row's bytes in
    pieces of P bytes; register slot i (8 bytes) is read from ring slot (i + li // 8) mod NS,
    NS = NT / 8 (whole 8-byte steps), then the words are rotated by one when bit 2 of li is
    set, then a funnel shift by 8 * (li & 3) bits."""
    NW, NS = NT // 4, NT // 8
    ring = list(stream_bytes)                              # piece q holds bytes q*P .. q*P+P-1
    regs = []
    for i in range(NS):
        j = (i + (li >> 3)) & (NS - 1)
        piece, off = (j * 8) // P, (j * 8) % P
        regs += ring[piece * P + off:piece * P + off + 8]
    r = [int.from_bytes(bytes(regs[4 * k:4 * k + 4]), "little") for k in range(NW)]
    if (li >> 2) & 1:
        r = [r[(k + 1) % NW] for k in range(NW)]
    sh = 8 * (li & 3)
    if sh:
        r = [((r[k] >> sh) | (r[(k + 1) % NW] << (32 - sh))) & 0xFFFFFFFF for k in range(NW)]
    return b"".join(w.to_bytes(4, "little") for w in r)


def test_slot_reads_are_conflict_free():
    """Each 8-byte slot read of a warp (ring layout [piece][thread][P bytes]) touches every bank
    pair at most twice: two wavefronts, the least 32 lanes x 8 bytes can take."""
    for NT, P in ((32, 16), (32, 8), (16, 16), (16, 8), (8, 8)):
        NS = NT // 8
        for i in range(NS):
            banks = {}
            for lane in range(32):
                li = lane % NT
                j = (i + (li >> 3)) & (NS - 1)
                addr = (j * 8 // P) * 1024 * P + lane * P + (j * 8) % P
                for w in range(2):
                    b = (addr // 4 + w) % BANKS
                    banks[b] = banks.get(b, 0) + 1
            assert max(banks.values()) <= 2, (NT, P, i)


@pytest.mark.parametrize("TP,M", [(1, 1), (1, 2), (1, 4), (2, 1), (2, 2), (2, 4), (4, 1),
                                  (4, 2), (4, 4)])
def test_rotation_brings_byte_s_plus_li_to_position_s(TP, M):
    """After the rotation, byte s of the lane's words is stream byte (s + li) mod NT -- the code
    of table (l' + s) mod NT that step s looks up -- for every lane and every instantiation's
    piece size P = min(NT, 8*M, 16)."""
    NT = 32 // TP
    P = min(min(NT, 8 * M), 16)
    stream = [(7 * i + 3) & 0xFF for i in range(NT)]
    for li in range(NT):
        rot = _kernel_rotation(stream, li, NT, P)
        assert list(rot) == [stream[(s + li) % NT] for s in range(NT)], (TP, M, li)
