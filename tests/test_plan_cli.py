"""Command-line planner: calibration arrays in, plan file out, the same plan as the library call
(no GPU)."""
import numpy as np
import pytest

import workloads as W


def _calib(n_layers=2):
    cfg = W.CONFIGS["tiny"]
    ks, vs, qs = [], [], []
    for layer in range(n_layers):
        ck, cv, cq = W.layer_calibration(cfg, layer, n=1024)
        ks.append(ck)
        vs.append(cv)
        qs.append(cq)
    return np.stack(ks), np.stack(vs), np.stack(qs)


def test_cli_writes_the_library_plan(aatc, tmp_path, capsys):
    from paper_2608_14191_gb300 import plan_cli
    k, v, q = _calib()
    npz = str(tmp_path / "calib.npz")
    np.savez(npz, k=k, v=v, q=q)
    out = str(tmp_path / "plan.aatc")
    assert plan_cli.main([npz, out, "--bits", "2.75"]) == 0
    assert "352 bits" in capsys.readouterr().out
    dm, p = aatc.load_plan(out)
    want = aatc.calibrate(aatc.dims(2, 1, 4), k, v, q, 2.75)
    for key in ("basis", "bits", "scales"):
        assert np.array_equal(p[key], want[key].reshape(p[key].shape)), key
    # the global pool over both layers (none protected) keeps the total budget
    out2 = str(tmp_path / "global.aatc")
    assert plan_cli.main([npz, out2, "--bits", "2.0", "--global", "--protect", "0"]) == 0
    _, pg = aatc.load_plan(out2)
    assert int(pg["bits"][:, :, 0].astype(int).sum()) == 2 * 256 and int(pg["bits"][:, :, 1].astype(int).sum()) == 2 * 256


def test_cli_without_queries_and_bad_shapes(aatc, tmp_path):
    from paper_2608_14191_gb300 import plan_cli
    k, v, _ = _calib(1)
    npz = str(tmp_path / "kv.npz")
    np.savez(npz, k=k, v=v)
    out = str(tmp_path / "p.aatc")
    assert plan_cli.main([npz, out, "--bits", "3", "--var-only", "--b-max", "16"]) == 0
    dm, p = aatc.load_plan(out)
    assert dm.b_max == 16 and int(p["bits"].astype(int).sum()) == 2 * 384
    with pytest.raises(ValueError):
        plan_cli.plan_from_arrays(k[..., :64], v[..., :64], None, 2.0, 2.0)
