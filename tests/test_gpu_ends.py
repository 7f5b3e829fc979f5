"""GPU parity of the network's ends through the C ABI, bit-exact against the CPU oracle: the first
layer on 8-bit image values (binary filters, integrated conversion to 2-bit codes) and the separated
fixed-point output of the detection conv (Sec. 2.2), alone and in the whole IFQ-Tinier-YOLO stack."""
import numpy as np
import pytest
import torch
from stack_parity import compare_stack_with_oracle

from oracle import oracle as O
from paper_1911_08076_gb300 import ifq, synth
from paper_1911_08076_gb300.stack import DeviceStack

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

DEV = "cuda"

IN8_CASES = [
    # B, H, W, C, cout, k, stride, pad, pool
    (2, 20, 20, 4, 8, 3, 1, 1, 0),        # RGB + zero channel: 4-byte pixels
    (2, 20, 20, 4, 8, 3, 1, 1, 2),        # with the fused 2x2 pool
    (1, 13, 11, 16, 32, 3, 2, 1, 0),      # 16-byte pixels, stride 2, ragged M
    (3, 9, 9, 20, 64, 3, 1, 1, 0),        # 20-byte pixels
    (2, 12, 12, 8, 16, 5, 1, 2, 0),       # 5x5 window
    (2, 17, 19, 4, 16, 3, 1, 1, 0),       # RGB first layer, 16 channels, odd sizes
    (2, 18, 18, 4, 12, 3, 1, 1, 2),       # 12 channels, fused pool
    (1, 10, 10, 4, 8, 3, 1, 0, 2),        # no padding, fused pool
]


@pytest.mark.parametrize("path", [ifq.IFQ_PATH_TC, ifq.IFQ_PATH_DIRECT], ids=["tc", "direct"])
@pytest.mark.parametrize("case", IN8_CASES, ids=[str(c) for c in IN8_CASES])
def test_conv_on_8bit_values_matches_oracle(case, path):
    B, H, W, C, cout, k, s, p, pool = case
    rng = np.random.default_rng(abs(hash(case)) % (2 ** 32))
    x = rng.integers(0, 256, (B, H, W, C), dtype=np.uint8)
    w = np.where(rng.integers(0, 2, (cout, k, k, C)) == 1, 1, -1).astype(np.int8)
    K = k * k * C
    K_fold = -(-255 * K // 3)
    sd = np.sqrt(K * 21717.0)                        # spread of A for uniform bytes and +-1 filters
    prm = O.Params(rng.uniform(0.5, 1.5, cout) * 3.0 / (sd * synth.PIXEL_STEP), rng.normal(1.0, 0.6, cout),
                   rng.normal(0, 0.5, cout), rng.normal(0, 1.0, cout), rng.uniform(0.5, 2.0, cout), None,
                   synth.PIXEL_STEP, 0.5, -0.25, synth.EPS)
    mode = ifq.IFQ_OUT_CODES if pool else ifq.IFQ_OUT_BOTH
    d = ifq.conv_desc(B, H, W, C, cout, k, s, p, mode, path, pool=pool, in_bits=8)
    direct_ok = cout <= 32 and K <= 257
    assert ifq.ifq_conv_plan(d) == (path if (path == ifq.IFQ_PATH_TC or direct_ok) else ifq.IFQ_PATH_TC)
    T, sg = ifq.ifq_fold_layer(K_fold, prm.alpha, prm.gamma, prm.beta, prm.mean, prm.var, prm.delta_in, None,
                               prm.eps, prm.q_base, prm.q_offset)
    bits = torch.from_numpy(synth.pack_signs(w).view(np.int32)).to(DEV)
    prep = torch.empty(ifq.ifq_weights_prep_bytes(d), dtype=torch.uint8, device=DEV)
    ifq.ifq_pack_weights(d, bits, prep)
    ho, wo = ifq.ifq_conv_out_shape(d)
    yc = torch.full((B, ho, wo, cout // 4), 0x5A, dtype=torch.uint8, device=DEV)
    ya = torch.full((B, ho, wo, cout), -777777, dtype=torch.int32, device=DEV) if not pool else None
    ifq.ifq_conv2bit(d, torch.from_numpy(x).to(DEV), prep, torch.from_numpy(T).to(DEV),
                     torch.from_numpy(sg).to(DEV), yc, ya)
    torch.cuda.synchronize()
    assert ifq.ifq_device_status() == ifq.IFQ_OK
    A = O.conv_acc(x, w, s, p)
    To, so = O.fold(prm, K_fold)
    if pool:
        ref = O.int_chain(O.maxpool_acc(A, pool, pool, 0), To, so)
    else:
        assert (ya.cpu().numpy() == A).all()
        ref, _ = O.check_chains(A, prm, To, so)
        assert len(np.unique(ref)) == 4
    assert (synth.unpack_codes(yc.cpu().numpy(), cout) == ref).all()


@pytest.mark.parametrize("m", [9, 14, 24])
def test_fixed_output_matches_oracle(m):
    rng = np.random.default_rng(m + 7)
    rows, cout = 3 * 169, 30
    alpha = rng.uniform(0.001, 0.5, cout).astype(np.float32)
    bias = rng.normal(0, 1, cout).astype(np.float32)
    A = rng.integers(-40000, 40000, (rows, cout)).astype(np.int32)
    A[0, :] = 2 ** 31 - 1                            # saturates at every m
    A[1, :] = -2 ** 31
    mul, add = ifq.ifq_fold_output_separated(m, alpha, synth.STEP, bias)
    y = torch.full((rows, cout), 12345, dtype=torch.int32, device=DEV)
    ifq.ifq_fixed_output(torch.from_numpy(A).to(DEV), rows, cout, torch.from_numpy(mul).to(DEV),
                         torch.from_numpy(add).to(DEV), m, y)
    ifq.ifq_fixed_output(torch.from_numpy(A).to(DEV), 0, cout, torch.from_numpy(mul).to(DEV),
                         torch.from_numpy(add).to(DEV), m, y)    # empty: nothing written
    torch.cuda.synchronize()
    p = O.Params(alpha.astype(np.float64), np.ones(cout), np.zeros(cout), np.zeros(cout), np.ones(cout),
                 bias.astype(np.float64), synth.STEP, 0.5, -0.25, 0.0)
    assert (y.cpu().numpy() == O.fixed_output(A, p, m)).all()


@pytest.mark.parametrize("name,batch", [("tinieryolo_full", 3), ("tinieryolo_full", 64)])
def test_tinier_yolo_full_matches_oracle(name, batch):
    """The whole IFQ-Tinier-YOLO stack with separate pool launches from 8-bit pixels to fixed-point
    detection outputs (the fused form is in the full-size workload tests); the oracle recomputes
    every image through every layer."""
    wl = synth.get(name, batch)
    x, params = synth.draw_workload(wl)
    compare_stack_with_oracle(wl, x, params)
